// dard_attention.cu - state-masked bidirectional attention of one DARD step (sm_103a).
//
// The augmented sequence x~_t = (x_t; s_t) of arXiv 2608.26574 Sec. 3.1 is stored per
// sequence as N original rows followed by S shadow rows. Every query attends exactly one
// copy (x^j or s^j) of every original position j (Eq. 2); which copy is decided in-kernel
// from the block's state vector and c_{t-1} (Sec. 3.2, query blocks 1-6 and Eq. 3). Key
// tiles that touch neither the current block nor the shadow rows are dense for every query,
// so the mask is evaluated only on the (at most three) tiles that contain block keys,
// shadow keys or the ragged end of the sequence.
//
// bf16 paths (tcgen05 MMAs with fp32 accumulators in TMEM, K/V tiles of 128 keys by TMA),
// one CTA per SM, chosen per call by a cost model (launch_tc):
//
// attn_tc1: 128 query rows of one (sequence, head); 11 warps:
//   warps 0-7  softmax and epilogue: warps w and w + 4 share TMEM lane quarter w (query
//              rows 32w .. 32w + 31), each taking 64 of a tile's 128 key columns;
//   warp 8     TMA producer: K and V through 3 stages each;
//   warp 9     TMEM allocator and PV issuer: O += P_j V_j, P_j (bf16) read from TMEM;
//   warp 10    S issuer: S_j = Q K_j^T (Q from TMEM, K from shared memory) into a ring of
//              two 128-column TMEM buffers, reused once the softmax has read S_j.
//   TMEM: S ring [0, 256), O [256, 256 + D), P [384, 448), Q [448, 448 + D/2). The
//   softmax threads write their query rows into TMEM at the start, so shared-memory
//   bandwidth goes to K and V only.
//
// attn_tc2: two 128-row query tiles of the same (sequence, head), so that every K/V tile
// serves 256 rows; 12 warps (warp 11 spare: it completes the side warpgroup's register split):
//   warps 4q .. 4q + 3  softmax and epilogue of tile q, one thread per query row;
//   warp 8              TMA producer: both Q tiles, then K and V through 2 stages each;
//   warp 9              TMEM allocator and S issuer: S_q(j) = Q_q K(j)^T (Q from shared
//                       memory), once PV_q(j - 1) has read P_q(j - 1) out of S_q's columns;
//   warp 10             PV issuer: O_q += P_q(j) V(j), each 64-key half as soon as that half
//                       of P_q(j) is stored.
//   TMEM: S_0, S_1 [0, 256) with P_q(j) written over the first 64 columns of S_q(j),
//   O_0, O_1 [256, 256 + 2D).
// Both keep a per-row running maximum and rescale O in TMEM only when the maximum grows by
// more than a factor 2^8 (the exponentials stay bounded by 2^8 otherwise).
// fp32 path: attn_simt (dard_attention_simt.cu), CUDA cores, the same mask logic.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <numeric>
#include <vector>

#include "dard_attn_common.cuh"

namespace dard {
namespace {

constexpr int kTc1Threads = 352;  // attn_tc1: 8 softmax warps, producer, PV issuer, S issuer
constexpr int kTc2Threads = 384;  // attn_tc2: 2 x 4 softmax warps, TMA producer, S and PV issuers, spare

constexpr int kQT = 2;   // query tiles per CTA (the same sequence and head)
constexpr int kNK = 2;   // TMA stages for K
constexpr int kNV = 2;   // TMA stages for V
constexpr int kWProd = 2 * kQT * 2;  // warp 8: TMA producer
constexpr int kWMma = kWProd + 1;    // warp 9: TMEM allocator and S issuer
constexpr int kWPv = kWProd + 2;     // warp 10: PV issuer
// attn_tc2 register split (setmaxnreg): the launch gives 384 threads 168 registers each; the
// warpgroup of warps 8-11 (producer, issuers, spare) drops to 56 and the two softmax
// warpgroups rise to 224, so that a thread holds its row's 128 scores at once:
// 128 x 56 + 256 x 224 = 384 x 168.
constexpr uint32_t kTc2LaunchRegs = 168, kTc2SideRegs = 56, kTc2SoftmaxRegs = 224;
static_assert(128 * kTc2SideRegs + 256 * kTc2SoftmaxRegs == kTc2Threads * kTc2LaunchRegs,
              "the register shares must add up to the launch's registers");
static_assert(kTc2Threads * kTc2LaunchRegs <= 65536, "one CTA per SM");

// Named barriers: 0 = __syncthreads, 1 = warps 0-3 (block info), 2 = the 8 softmax warps,
// then per kernel: attn_tc1 3 + q = the two warps sharing TMEM lane quarter q; attn_tc2
// 3 + q = the four warps of query tile q.
__device__ __forceinline__ void tile_bar_sync(int q) {
  asm volatile("bar.sync %0, 128;" ::"r"(3 + q) : "memory");
}

constexpr int kNS = 2;   // S buffers in TMEM (a ring of 128-column buffers)
constexpr int kNKV = 3;  // TMA stages for K and for V
constexpr int kSoftmaxWarps = 8;  // two warps per query row, 64 key columns each

// Every barrier completes one phase per use of its ring slot; tile j uses slot j % ring
// and waits for parity (j / ring) & 1. A waiter is never more than one phase behind the
// phase it waits for (the parity would alias otherwise): each wait for use u of a slot is
// preceded, in the same thread or through a chain of waits, by the completion of use u - 1.
struct __align__(16) Tc1Ctl {
  uint64_t q_full, o_full, p_full, pv_done;
  uint64_t k_full[kNKV], k_empty[kNKV], v_full[kNKV], v_empty[kNKV];
  uint64_t s_full[kNS], s_free[kNS];
  uint64_t drained;  // every product both issuers launched has completed (two commits)
  uint32_t tmem_base;
  int32_t abort;
  BlockInfo bi;
  float red_max[2][2][kBM];  // per tile (double-buffered by tile parity): the two column
                             // halves' row maxima
  float red_sum[2][kBM];   // at the end: the two halves' row sums
  uint8_t store_row[kBM];  // epilogue: rows of this tile that are written
};

template <int D>
constexpr size_t tc1_smem_bytes() {
  // alignment slack + kNKV stages each of K and V (128 rows) + control
  return 1024 + 2 * kNKV * static_cast<size_t>(kTN) * D * 2 + sizeof(Tc1Ctl);
}

__device__ __forceinline__ void flag_timeout(const AttnParams& p, Tc1Ctl& ctl) {
  ctl.abort = 1;
  if (p.status) atomicOr(p.status, DARD_STATUS_TIMEOUT);
}

template <int D>
__global__ void __launch_bounds__(kTc1Threads, 1)
    attn_tc1(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tmk,
            const __grid_constant__ CUtensorMap tmv) {
  constexpr int kSub = D / 64;                 // 128-byte (64 x bf16) column blocks
  constexpr uint32_t kKSub = kTN * 128;        // one 128-row x 128-byte swizzled block
  constexpr uint32_t kKVBytes = kSub * kKSub;  // one K (or V) tile of 128 keys
  constexpr int kWProd = kSoftmaxWarps, kWPV = kSoftmaxWarps + 1, kWS = kSoftmaxWarps + 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = base;                  // kNKV stages
  uint8_t* sV = sK + kNKV * kKVBytes;  // kNKV stages
  Tc1Ctl& ctl = *reinterpret_cast<Tc1Ctl*>(sV + kNKV * kKVBytes);

  int seq, qt, h;
  decode_work(p, blockIdx.x, seq, qt, h);
  const SeqDesc sd = p.seq[seq];
  const int rows_seq = sd.n_orig + sd.slen;
  const int q0 = sd.q_start + qt * kBM;  // first (sequence-relative) query row of the tile
  const int n_kt = key_tiles(sd, q0, min(q0 + kBM, rows_seq));  // shadow-only tiles skipped
  const int g = h / (p.hq / p.hkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long wlim = p.wait_cycles > 0 ? p.wait_cycles : kWaitCycles;

  // The producer lane initialises the barriers and issues the first kNKV K/V tiles at
  // once; the other threads touch the barriers only after the block-wide sync below.
  const int row0 = sd.row_base;
  auto load_kv = [&](int j, bool k_or_v) {
    const int b = j % kNKV;
    uint64_t* bar = k_or_v ? &ctl.k_full[b] : &ctl.v_full[b];
    uint8_t* dst = (k_or_v ? sK : sV) + b * kKVBytes;
    const void* map = k_or_v ? static_cast<const void*>(&tmk) : static_cast<const void*>(&tmv);
    mbar_arrive_expect_tx(bar, kKVBytes);
    if (k_or_v && j == p.test_drop_kv) return;  // test hook: this K copy is never issued
#pragma unroll
    for (int s = 0; s < kSub; ++s)
      tma_load_2d(dst + s * kKSub, map, bar, g * D + s * 64, row0 + j * kTN);
  };
  if (warp == kWProd && lane == 0) {
    mbar_init(&ctl.q_full, kSoftmaxWarps);  // each softmax warp writes half of its Q rows
    mbar_init(&ctl.drained, 2);
    mbar_init(&ctl.o_full, 1);
    mbar_init(&ctl.p_full, kSoftmaxWarps);
    mbar_init(&ctl.pv_done, 1);
    for (int b = 0; b < kNKV; ++b) {
      mbar_init(&ctl.k_full[b], 1);
      mbar_init(&ctl.k_empty[b], 1);
      mbar_init(&ctl.v_full[b], 1);
      mbar_init(&ctl.v_empty[b], 1);
    }
    for (int b = 0; b < kNS; ++b) {
      mbar_init(&ctl.s_full[b], 1);
      mbar_init(&ctl.s_free[b], kSoftmaxWarps);
    }
    ctl.abort = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmk);
    tma_prefetch_desc(&tmv);
    grid_dep_wait();  // the RoPE key pass launched before this kernel (if any) is complete
    for (int j = 0; j < kNKV && j < n_kt; ++j) {
      load_kv(j, true);
      load_kv(j, false);
    }
  }
  if (warp == kWPV) {
    tmem_alloc<kTmemCols>(&ctl.tmem_base);
    tmem_relinquish();
  }
  // Softmax warp w: rows 32 (w % 4) .. + 31 (TMEM lane quarter), key columns 64 (w / 4) ..
  const int quarter = warp & 3, half = warp >> 2;
  const int t = quarter * 32 + lane;  // this thread's query row within the tile
  BlockFetch bf{-1, 0.f, -1};
  uint4 qhalf[D / 16];  // half of this thread's query row (bf16)
  if (warp < kSoftmaxWarps) {
    if (half == 0) bf = fetch_block_info(p, sd);  // in flight across the block sync
    const int r = row0 + q0 + t;
    const uint4* src = reinterpret_cast<const uint4*>(
        static_cast<const __nv_bfloat16*>(p.q) + (static_cast<size_t>(r) * p.hq + h) * D +
        half * (D / 2));
#pragma unroll
    for (int c = 0; c < D / 16; ++c)
      qhalf[c] = r < p.total_rows ? __ldg(src + c) : make_uint4(0, 0, 0, 0);
    if (p.rope && q0 + t < rows_seq) {  // RoPE of this row (rows of the next sequence: unused)
      const int pos = rope_position(p, sd, q0 + t);
      if (p.rope_style == DARD_ROPE_INTERLEAVED) {
#pragma unroll
        for (int c = 0; c < D / 16; ++c)
          rope_chunk_interleaved(qhalf[c], pos, p.rope_f + 8 * (half * (D / 16) + c));
      } else {  // the partner of each element is at the same offset of the other half
        const uint4* other = src + (half == 0 ? D / 16 : -(D / 16));
#pragma unroll
        for (int c = 0; c < D / 16; ++c)
          rope_chunk_half(qhalf[c], __ldg(other + c), half == 0, pos, p.rope_f + 16 * c);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // TMEM columns: S ring [0, 256), O [256, 256 + D), P [384, 448), Q [448, 448 + D / 2)
  const uint32_t tO = ctl.tmem_base + kNS * kTN;
  const uint32_t tP = ctl.tmem_base + 384;
  const uint32_t tQ = ctl.tmem_base + 448;
  volatile int32_t* abort_flag = &ctl.abort;

  if (warp == kWProd) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int last_k = min(n_kt, kNKV) - 1, last_v = last_k;
      for (int j = kNKV; j < n_kt && !*abort_flag; ++j) {
        const int b = j % kNKV, ph = ((j - kNKV) / kNKV) & 1;
        if (!mbar_wait(&ctl.k_empty[b], ph, wlim)) { flag_timeout(p, ctl); break; }
        load_kv(j, true);
        last_k = j;
        if (!mbar_wait(&ctl.v_empty[b], ph, wlim)) { flag_timeout(p, ctl); break; }
        load_kv(j, false);
        last_v = j;
      }
      {
        // Every copy issued lands before shared memory is released (after a normal run they
        // all have: the waits return at once): the latest use of each stage (earlier uses
        // landed before their stage was reused). A copy the test hook dropped was never
        // issued.
        for (int b = 0; b < kNKV; ++b) {
          const int jk = last_k - ((last_k - b) % kNKV + kNKV) % kNKV;
          const int jv = last_v - ((last_v - b) % kNKV + kNKV) % kNKV;
          if (last_k >= 0 && jk >= 0 && jk != p.test_drop_kv)
            mbar_wait(&ctl.k_full[b], (jk / kNKV) & 1, wlim);
          if (last_v >= 0 && jv >= 0) mbar_wait(&ctl.v_full[b], (jv / kNKV) & 1, wlim);
        }
      }
    }
  } else if (warp == kWS) {
    // ------------------------------------------------------------ S issuer
    // S_t = Q K_t^T (Q from TMEM, K from shared memory) into ring buffer t % kNS as soon as
    // K_t has landed and the softmax has read S_{t - kNS} out of that buffer.
    if (lane == 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(kBM, kTN, 0, 0);
      const uint32_t ak = smem_u32(sK);
      bool ok = mbar_wait(&ctl.q_full, 0, wlim);
      for (int t2 = 0; t2 < n_kt && ok && !*abort_flag; ++t2) {
        const int kb = t2 % kNKV, sb = t2 % kNS;
        if (t2 >= kNS) ok = mbar_wait(&ctl.s_free[sb], ((t2 - kNS) / kNS) & 1, wlim);
        ok = ok && mbar_wait(&ctl.k_full[kb], (t2 / kNKV) & 1, wlim);
        if (!ok) break;
        tc_fence_after();
        const uint32_t kaddr = ak + kb * kKVBytes;
        const uint32_t dst = ctl.tmem_base + sb * kTN;
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t ko = (ks >> 2) * kKSub + (ks & 3) * 32;
          mma_ts(dst, tQ + ks * 8, smem_desc_sw128(kaddr + ko, 16, 1024), kIdS, ks > 0);
        }
        mma_commit(&ctl.s_full[sb]);
        mma_commit(&ctl.k_empty[kb]);
      }
      if (!ok) flag_timeout(p, ctl);
      mma_commit(&ctl.drained);  // completes once every S product this thread issued has
    }
  } else if (warp == kWPV) {
    // ------------------------------------------------------------ PV issuer
    // O += P_j V_j as soon as the softmax has written P_j and V_j has landed.
    if (lane == 0) {
      constexpr uint32_t kIdO = idesc_bf16_f32(kBM, D, 0, 1);
      const uint32_t av = smem_u32(sV);
      bool ok = true;
      for (int j = 0; j < n_kt && ok && !*abort_flag; ++j) {
        const int vb = j % kNKV;
        ok = mbar_wait(&ctl.p_full, j & 1, wlim) && mbar_wait(&ctl.v_full[vb], (j / kNKV) & 1, wlim);
        if (!ok) break;
        tc_fence_after();
        const uint32_t vaddr = av + vb * kKVBytes;
#pragma unroll
        for (int ks = 0; ks < kTN / 16; ++ks)
          mma_ts(tO, tP + ks * 8, smem_desc_sw128(vaddr + ks * 2048, kKSub, 1024), kIdO,
                 (j > 0 || ks > 0) ? 1u : 0u);
        mma_commit(&ctl.pv_done);
        mma_commit(&ctl.v_empty[vb]);
        if (j == n_kt - 1) mma_commit(&ctl.o_full);
      }
      if (!ok) flag_timeout(p, ctl);
      mma_commit(&ctl.drained);  // completes once every PV product this thread issued has
    }
  } else {
    // ------------------------------------------------------------ softmax + epilogue
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    {  // this warp's half of the query rows into TMEM (bf16 pairs, the A-operand layout)
#pragma unroll
      for (int c = 0; c < D / 128; ++c) {
        uint32_t w[32];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          w[4 * e + 0] = qhalf[8 * c + e].x;
          w[4 * e + 1] = qhalf[8 * c + e].y;
          w[4 * e + 2] = qhalf[8 * c + e].z;
          w[4 * e + 3] = qhalf[8 * c + e].w;
        }
        tmem_st32(tQ + lane_off + half * (D / 4) + 32 * c, w);
      }
      if (D == 64) {  // 16 columns per half
        uint32_t w[16];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          w[4 * e + 0] = qhalf[e].x;
          w[4 * e + 1] = qhalf[e].y;
          w[4 * e + 2] = qhalf[e].z;
          w[4 * e + 3] = qhalf[e].w;
        }
        tmem_st16(tQ + lane_off + half * 16, w);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.q_full);
    }
    if (half == 0) publish_block_info(p, sd, ctl.bi, bf, qt == 0 && h == 0);
    softmax_bar_sync();
    const RowInfo q = row_info(sd, ctl.bi, q0 + t);
    const RowMasks rm = row_masks(q, ctl.bi, sd);
    const float sl = p.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < n_kt; ++j) {
      const int b = j % kNS;
      const int kt0 = j * kTN + half * 64;  // this warp's 64 keys
      const bool masked = tile_needs_mask(sd, j * kTN);
      const uint64_t vis = masked ? vis64(sd, kt0, rm) : ~0ull;
      // Both warps of the rows wait for the same S_j with the same bound (no early leave on
      // an abort flag), so they leave the loop together: a barrier completing between the two
      // warps' deadlines (a product about a second late) is the only way they could part.
      ok = mbar_wait(&ctl.s_full[b], (j / kNS) & 1, wlim);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      float s[64];
      {
        uint32_t r0[32], r1[32];
        tmem_ld32(ctl.tmem_base + b * kTN + 64 * half + lane_off, r0);
        tmem_ld32(ctl.tmem_base + b * kTN + 64 * half + 32 + lane_off, r1);
        tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          s[e] = __uint_as_float(r0[e]);
          s[32 + e] = __uint_as_float(r1[e]);
        }
      }
      // S_j is in registers: the S issuer may reuse its buffer
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.s_free[b]);
      if (masked) {
#pragma unroll
        for (int k = 0; k < 64; ++k) s[k] = ((vis >> k) & 1ull) ? s[k] : -INFINITY;
      }
      float mx[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = fmax3(s[e], s[8 + e], s[16 + e]);
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = fmax3(mx[e], s[24 + e], s[32 + e]);
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = fmax3(mx[e], s[40 + e], s[48 + e]);
#pragma unroll
      for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], s[56 + e]);
      const float mh = fmaxf(fmax3(mx[0], mx[1], mx[2]),
                             fmax3(fmax3(mx[3], mx[4], mx[5]), mx[6], mx[7]));
      ctl.red_max[j & 1][half][t] = mh;
      pair_bar_sync(quarter);
      const float mt = fmaxf(mh, ctl.red_max[j & 1][half ^ 1][t]);
      // Raise the reference maximum on the first finite value, or when the tile maximum
      // exceeds it by more than 2^kRescaleLog2 in probability; only then is O rescaled.
      // Both warps of a row take the same decision from the same values.
      float m_new = m_run;
      if (m_run == -INFINITY) m_new = mt;
      else if ((mt - m_run) * sl > kRescaleLog2) m_new = mt;
      const bool rescale = (m_new != m_run) && (m_run != -INFINITY);
      const float alpha = rescale ? ex2_approx((m_run - m_new) * sl) : 1.f;
      const float mL = (m_new == -INFINITY) ? 0.f : m_new * sl;
      uint32_t pk[32];
      const uint64_t sl2 = f2_pack(sl, sl), nmL2 = f2_pack(-mL, -mL);
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};  // partial sums
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        float x0, x1;
        f2_unpack(f2_fma(f2_pack(s[2 * e], s[2 * e + 1]), sl2, nmL2), x0, x1);
        pk[e] = pack_bf16x2(ex2_approx(x0), ex2_approx(x1));
        // the row sum adds the rounded weights the PV product multiplies with (two
        // mixed-precision adds: faster here than unpacking into a packed pair)
        add_bf16x2_f32(acc[2 * (e & 3)], acc[2 * (e & 3) + 1], pk[e]);
      }
      float ls[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) ls[k] = acc[k] + acc[4 + k];
      // P_j replaces P_{j-1}, and O may be rescaled, once PV_{j-1} has completed
      if (j > 0) {
        ok = mbar_wait(&ctl.pv_done, (j - 1) & 1, wlim);  // the same barrier for both warps
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after();
      }
      if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
        for (int c = 0; c < D / 64; ++c) {  // this warp's half of the O columns
          uint32_t r[32];
          const uint32_t col = tO + lane_off + half * (D / 2) + 32 * c;
          tmem_ld32(col, r);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
          tmem_st32(col, r);
        }
      }
      l_run = l_run * alpha + ((ls[0] + ls[1]) + (ls[2] + ls[3]));
      m_run = m_new;
      tmem_st32(tP + lane_off + 32 * half, pk);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.p_full);
    }
    if (ok) ok = mbar_wait(&ctl.o_full, 0, wlim);
    const bool wok = __all_sync(0xffffffffu, ok);
    if (!wok && lane == 0) flag_timeout(p, ctl);
    // O row / row sum -> bf16 into shared memory (the K stages are no longer read once
    // o_full has completed), 16-byte chunks XOR-swizzled by row; then the 256 softmax
    // threads store whole rows, coalesced. Every softmax warp reaches the named barriers
    // on every path.
    ctl.red_sum[half][t] = l_run;
    softmax_bar_sync();
    constexpr int kChunks = D / 8;  // 16-byte chunks per output row
    const int r = q0 + t;
    uint4* stage = reinterpret_cast<uint4*>(sK);  // 128 rows x D bf16 <= one K stage
    if (wok) {
      tc_fence_after();
      const float inv_l = 1.0f / (ctl.red_sum[0][t] + ctl.red_sum[1][t]);
#pragma unroll
      for (int c = 0; c < D / 64; ++c) {
        uint32_t rr[32];
        tmem_ld32(tO + lane_off + half * (D / 2) + 32 * c, rr);
        tmem_wait_ld();
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          uint4 u;
          u.x = pack_bf16x2(__uint_as_float(rr[8 * v + 0]) * inv_l, __uint_as_float(rr[8 * v + 1]) * inv_l);
          u.y = pack_bf16x2(__uint_as_float(rr[8 * v + 2]) * inv_l, __uint_as_float(rr[8 * v + 3]) * inv_l);
          u.z = pack_bf16x2(__uint_as_float(rr[8 * v + 4]) * inv_l, __uint_as_float(rr[8 * v + 5]) * inv_l);
          u.w = pack_bf16x2(__uint_as_float(rr[8 * v + 6]) * inv_l, __uint_as_float(rr[8 * v + 7]) * inv_l);
          const int chunk = half * (kChunks / 2) + c * 4 + v;
          stage[t * kChunks + (chunk ^ (t & (kChunks - 1)))] = u;
        }
      }
    }
    if (half == 0) ctl.store_row[t] = (wok && q.store && r < rows_seq) ? 1 : 0;
    softmax_bar_sync();
    if (!*abort_flag) {
      __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.o);
      const int tid = threadIdx.x;  // 0 .. 255
#pragma unroll 4
      for (int idx = tid; idx < kBM * kChunks; idx += 32 * kSoftmaxWarps) {
        const int row = idx / kChunks, chunk = idx % kChunks;
        if (ctl.store_row[row]) {
          const uint4 u = stage[row * kChunks + (chunk ^ (row & (kChunks - 1)))];
          uint4* dst = reinterpret_cast<uint4*>(
              out + (static_cast<size_t>(sd.row_base + q0 + row) * p.hq + h) * D);
          dst[chunk] = u;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kWPV) {
    // no product is still writing TMEM (both issuers committed `drained` last)
    if (lane == 0 && !mbar_wait(&ctl.drained, 0, wlim)) flag_timeout(p, ctl);
    __syncwarp();
    tc_fence_after();
    tmem_dealloc<kTmemCols>(ctl.tmem_base);
  }
}


// One query row's 128-key S tile out of TMEM (columns tS .. tS + 127 of its lane) into
// registers, with the visibility bits applied (kMasked; vis0: keys 0-63, vis1: 64-127, a
// hidden key becomes -inf); returns the row maximum. One wait for the four loads.
template <bool kMasked>
__device__ __forceinline__ float tile_row_load(uint32_t tS, uint64_t vis0, uint64_t vis1,
                                               uint32_t (&sv)[128]) {
#pragma unroll
  for (int c = 0; c < 4; ++c) tmem_ld32(tS + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(sv + 32 * c));
  tmem_wait_ld();
  if (kMasked) {
#pragma unroll
    for (int k = 0; k < 128; ++k) {
      const uint64_t vis = k < 64 ? vis0 : vis1;
      sv[k] = ((vis >> (k & 63)) & 1ull) ? sv[k] : 0xff800000u;  // -inf
    }
  }
  float mx[8];
#pragma unroll
  for (int e = 0; e < 8; ++e)
    mx[e] = fmax3(__uint_as_float(sv[e]), __uint_as_float(sv[8 + e]), __uint_as_float(sv[16 + e]));
#pragma unroll
  for (int k = 24; k < 128; k += 16) {
#pragma unroll
    for (int e = 0; e < 8; ++e)
      mx[e] = k + 8 + e < 128 ? fmax3(mx[e], __uint_as_float(sv[k + e]), __uint_as_float(sv[k + 8 + e]))
                              : fmaxf(mx[e], __uint_as_float(sv[k + e]));
  }
  return fmaxf(fmax3(mx[0], mx[1], mx[2]), fmax3(fmax3(mx[3], mx[4], mx[5]), mx[6], mx[7]));
}

// P = 2^(s * sl - mL) for keys 64 hh .. 64 hh + 63 of the row's 128 scores held in
// registers, stored as bf16 pairs over columns tS + 32 hh .. tS + 32 hh + 31 (in the first
// half of the S tile's columns); the stored (rounded) values are summed into acc (four packed
// partial sums), so that the output is a convex combination of V rows with exactly the
// weights the PV product uses.
template <int hh>
__device__ __forceinline__ void tile_row_exp(uint32_t tS, const uint32_t (&sv)[128],
                                             uint64_t sl2, uint64_t nmL2, uint64_t (&acc)[4]) {
  {
    uint32_t pk[32];
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      float x0, x1;
      f2_unpack(f2_fma(f2_pack(__uint_as_float(sv[64 * hh + 2 * e]),
                               __uint_as_float(sv[64 * hh + 2 * e + 1])), sl2, nmL2), x0, x1);
      pk[e] = pack_bf16x2(ex2_approx(x0), ex2_approx(x1));
      // the row sum adds the rounded weights the PV product multiplies with (unpacked by
      // shift and mask into a packed pair: faster here than two mixed-precision adds)
      acc[e & 3] = f2_add(acc[e & 3], f2_pack(__uint_as_float(pk[e] << 16),
                                              __uint_as_float(pk[e] & 0xffff0000u)));
    }
    tmem_st32(tS + 32 * hh, pk);
  }
}

// Barrier protocol. Every barrier completes one phase per use; use u waits for parity
// (u / ring) & 1, and no waiter is ever two phases behind (the parity would alias):
// each wait for use u is preceded, in the same thread or through a chain of waits, by the
// completion of use u - ring.
struct __align__(16) Tc2Ctl {
  uint64_t q_full[kQT];  // query tile q landed
  uint64_t q_rot[kQT];   // RoPE: the softmax warps of tile q rotated it in shared memory
  uint64_t k_full[kNK], k_empty[kNK], v_full[kNV], v_empty[kNV];
  uint64_t s_full[kQT];   // S_q(j) landed in TMEM
  uint64_t p_half[kQT][2];  // the softmax of tile q stored keys 64 h .. 64 h + 63 of P_q(j)
  uint64_t pv_done[kQT];  // PV_q(j) completed: S_q's columns may take S_q(j + 1)
  uint64_t o_full[kQT];   // the last PV_q completed
  uint64_t drained;       // every product both issuers launched has completed (two commits)
  uint32_t tmem_base;
  int32_t abort;
  BlockInfo bi;
  uint8_t store_row[kQT][kBM];  // epilogue: rows of each tile that are written
};

template <int D>
constexpr size_t tc2_smem_bytes() {
  // alignment slack + kQT query tiles + kNK K stages + kNV V stages (128 rows each) + control
  return 1024 + (kQT + kNK + kNV) * static_cast<size_t>(kTN) * D * 2 + sizeof(Tc2Ctl);
}

__device__ __forceinline__ void flag_timeout(const AttnParams& p, Tc2Ctl& ctl) {
  ctl.abort = 1;
  if (p.status) atomicOr(p.status, DARD_STATUS_TIMEOUT);
}

// kRope: the launch applies RoPE to the query tiles (a separate instantiation, so that the
// kernel without RoPE keeps its register allocation).
template <int D, bool kRope>
__global__ void __launch_bounds__(kTc2Threads, 1)
    attn_tc2(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tmq,
            const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv) {
  constexpr int kSub = D / 64;                   // 128-byte (64 x bf16) column blocks
  constexpr uint32_t kKSub = kTN * 128;          // one 128-row x 128-byte swizzled block
  constexpr uint32_t kTileBytes = kSub * kKSub;  // one 128-row tile of Q, K or V
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = base;                     // kQT query tiles
  uint8_t* sK = sQ + kQT * kTileBytes;    // kNK stages
  uint8_t* sV = sK + kNK * kTileBytes;    // kNV stages
  Tc2Ctl& ctl = *reinterpret_cast<Tc2Ctl*>(sV + kNV * kTileBytes);

  int seq, pr, h;
  decode_pair(p, blockIdx.x, seq, pr, h);
  const SeqDesc sd = p.seq[seq];
  const int rows_seq = sd.n_orig + sd.slen;
  const int qt0 = kQT * pr;                       // first query tile of this CTA
  const int nq = min(kQT, sd.n_qtiles - qt0);     // 1 or 2 query tiles
  const int r0 = sd.q_start + qt0 * kBM;
  const int n_kt = key_tiles(sd, r0, min(r0 + nq * kBM, rows_seq));  // shadow-only tiles skipped
  const int g = h / (p.hq / p.hkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row0 = sd.row_base;
  const long long wlim = p.wait_cycles > 0 ? p.wait_cycles : kWaitCycles;

  auto load_kv = [&](int j, bool k_or_v) {
    const int b = j % (k_or_v ? kNK : kNV);
    uint64_t* bar = k_or_v ? &ctl.k_full[b] : &ctl.v_full[b];
    uint8_t* dst = (k_or_v ? sK : sV) + b * kTileBytes;
    const void* map = k_or_v ? static_cast<const void*>(&tmk) : static_cast<const void*>(&tmv);
    mbar_arrive_expect_tx(bar, kTileBytes);
    if (k_or_v && j == p.test_drop_kv) return;  // test hook: this K copy is never issued
#pragma unroll
    for (int s = 0; s < kSub; ++s)
      tma_load_2d(dst + s * kKSub, map, bar, g * D + s * 64, row0 + j * kTN);
  };
  auto load_q = [&](int q) {
    mbar_arrive_expect_tx(&ctl.q_full[q], kTileBytes);
#pragma unroll
    for (int s = 0; s < kSub; ++s)
      tma_load_2d(sQ + q * kTileBytes + s * kKSub, &tmq, &ctl.q_full[q], h * D + s * 64,
                  row0 + sd.q_start + (qt0 + q) * kBM);
  };
  // The producer lane initialises the barriers and issues Q0 and K0; the other threads touch
  // the barriers only after the block sync.
  if (warp == kWProd && lane == 0) {
    for (int q = 0; q < kQT; ++q) {
      mbar_init(&ctl.q_full[q], 1);
      mbar_init(&ctl.q_rot[q], 4);  // the tile's softmax warps
    }
    mbar_init(&ctl.drained, 2);
    for (int b = 0; b < kNK; ++b) {
      mbar_init(&ctl.k_full[b], 1);
      mbar_init(&ctl.k_empty[b], 1);
    }
    for (int b = 0; b < kNV; ++b) {
      mbar_init(&ctl.v_full[b], 1);
      mbar_init(&ctl.v_empty[b], 1);
    }
    for (int q = 0; q < kQT; ++q) {
      mbar_init(&ctl.s_full[q], 1);
      mbar_init(&ctl.p_half[q][0], 4);
      mbar_init(&ctl.p_half[q][1], 4);
      mbar_init(&ctl.pv_done[q], 1);
      mbar_init(&ctl.o_full[q], 1);
    }
    ctl.abort = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmq);
    tma_prefetch_desc(&tmk);
    tma_prefetch_desc(&tmv);
    // Q0 and K0 only: the first S product needs nothing else, and with every CTA of the
    // launch starting at once they land sooner alone (the rest follows in the producer)
    load_q(0);
    grid_dep_wait();  // the RoPE key pass launched before this kernel (if any) is complete
    load_kv(0, true);
  }
  if (warp == kWMma) {
    tmem_alloc<kTmemCols>(&ctl.tmem_base);
    tmem_relinquish();
  }
  BlockFetch bf{-1, 0.f, -1};
  if (warp < 4) bf = fetch_block_info(p, sd);  // in flight across the block sync
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // TMEM columns: S_q / P_q [128 q, 128 q + 128) (P_q(j) as bf16 pairs over the first 64),
  // O_q [256 + D q, 256 + D q + D)
  const uint32_t tS0 = ctl.tmem_base;
  const uint32_t tO0 = ctl.tmem_base + kQT * kTN;
  volatile int32_t* abort_flag = &ctl.abort;

  // The register split: each branch below starts with its warpgroup's setmaxnreg (warps 8-11
  // give registers up, the softmax warps 0-7 take them), so that it covers the branch's code.
  if (warp == kWProd) {
    // ------------------------------------------------------------ TMA producer
    reg_dealloc<kTc2SideRegs>();
    if (lane == 0) {
      // the other first loads once Q0 and K0 have landed
      int last_k = 0, last_v = -1, q_loaded = 1;
      if (!mbar_wait(&ctl.q_full[0], 0, wlim) || !mbar_wait(&ctl.k_full[0], 0, wlim)) {
        flag_timeout(p, ctl);
      } else {
        if (nq > 1) {
          load_q(1);
          q_loaded = 2;
        }
        load_kv(0, false);
        last_v = 0;
        for (int j = 1; j < kNK && j < n_kt; ++j) { load_kv(j, true); last_k = j; }
        for (int j = 1; j < kNV && j < n_kt; ++j) { load_kv(j, false); last_v = j; }
      }
      for (int j = min(kNK, kNV); j < n_kt && !*abort_flag; ++j) {
        if (j >= kNK) {
          const int b = j % kNK;
          if (!mbar_wait(&ctl.k_empty[b], ((j - kNK) / kNK) & 1, wlim)) { flag_timeout(p, ctl); break; }
          load_kv(j, true);
          last_k = j;
        }
        if (j >= kNV) {
          const int b = j % kNV;
          if (!mbar_wait(&ctl.v_empty[b], ((j - kNV) / kNV) & 1, wlim)) { flag_timeout(p, ctl); break; }
          load_kv(j, false);
          last_v = j;
        }
      }
      {
        // Every copy issued lands before shared memory is released (after a normal run they
        // all have: the waits return at once): the latest use of each stage (earlier uses
        // landed before their stage was reused). A copy the test hook dropped was never
        // issued.
        for (int b = 0; b < kNK; ++b) {
          const int jk = last_k - ((last_k - b) % kNK + kNK) % kNK;
          if (last_k >= 0 && jk >= 0 && jk != p.test_drop_kv)
            mbar_wait(&ctl.k_full[b], (jk / kNK) & 1, wlim);
        }
        for (int b = 0; b < kNV; ++b) {
          const int jv = last_v - ((last_v - b) % kNV + kNV) % kNV;
          if (last_v >= 0 && jv >= 0) mbar_wait(&ctl.v_full[b], (jv / kNV) & 1, wlim);
        }
        for (int q = 0; q < q_loaded; ++q) mbar_wait(&ctl.q_full[q], 0, wlim);
      }
    }
  } else if (warp == kWMma) {
    // ------------------------------------------------------------ S issuer
    reg_dealloc<kTc2SideRegs>();
    // S_q(j) = Q_q K(j)^T once K(j) has landed and, for j > 0, PV_q(j - 1) has completed
    // (S_q(j) overwrites the P_q(j - 1) that PV_q(j - 1) reads). The PV products come from
    // a second issuer thread: one thread issuing both kinds of product in turn leaves the
    // tensor pipe at about two thirds of its rate on this GPU.
    if (lane == 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(kBM, kTN, 0, 0);
      const uint32_t aq = smem_u32(sQ), ak = smem_u32(sK);
      bool ok = true;
      for (int j = 0; j < n_kt && ok && !*abort_flag; ++j) {
        ok = mbar_wait(&ctl.k_full[j % kNK], (j / kNK) & 1, wlim);
        for (int q = 0; q < nq && ok; ++q) {
          if (j == 0) ok = mbar_wait(kRope ? &ctl.q_rot[q] : &ctl.q_full[q], 0, wlim);
          else ok = mbar_wait(&ctl.pv_done[q], (j - 1) & 1, wlim);
          if (!ok) break;
          tc_fence_after();
          const uint32_t qaddr = aq + q * kTileBytes, kaddr = ak + (j % kNK) * kTileBytes;
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const uint32_t off = (ks >> 2) * kKSub + (ks & 3) * 32;
            mma_ss(tS0 + q * kTN, smem_desc_sw128(qaddr + off, 16, 1024),
                   smem_desc_sw128(kaddr + off, 16, 1024), kIdS, ks > 0);
          }
          mma_commit(&ctl.s_full[q]);
        }
        if (ok) mma_commit(&ctl.k_empty[j % kNK]);
      }
      if (!ok) flag_timeout(p, ctl);
      mma_commit(&ctl.drained);  // completes once every S product this thread issued has
    }
  } else if (warp == kWPv) {
    // ------------------------------------------------------------ PV issuer
    reg_dealloc<kTc2SideRegs>();
    // O_q += P_q(j) V(j) once V(j) has landed, in two halves of 64 keys: each as soon as
    // the softmax of tile q has stored that half of P_q(j), so that the first half's
    // products run while the softmax computes the second.
    if (lane == 0) {
      constexpr uint32_t kIdO = idesc_bf16_f32(kBM, D, 0, 1);
      const uint32_t av = smem_u32(sV);
      bool ok = true;
      for (int j = 0; j < n_kt && ok && !*abort_flag; ++j) {
        ok = mbar_wait(&ctl.v_full[j % kNV], (j / kNV) & 1, wlim);
        for (int q = 0; q < nq && ok; ++q) {
          const uint32_t vaddr = av + (j % kNV) * kTileBytes;
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            ok = ok && mbar_wait(&ctl.p_half[q][hh], j & 1, wlim);
            if (!ok) break;
            tc_fence_after();
#pragma unroll
            for (int ks = 4 * hh; ks < 4 * hh + 4; ++ks)
              mma_ts(tO0 + q * D, tS0 + q * kTN + ks * 8,
                     smem_desc_sw128(vaddr + ks * 2048, kKSub, 1024), kIdO,
                     (j > 0 || ks > 0) ? 1u : 0u);
          }
          if (!ok) break;
          mma_commit(&ctl.pv_done[q]);
          if (j == n_kt - 1) mma_commit(&ctl.o_full[q]);
        }
        if (ok) mma_commit(&ctl.v_empty[j % kNV]);
      }
      if (!ok) flag_timeout(p, ctl);
      mma_commit(&ctl.drained);  // completes once every PV product this thread issued has
    }
  } else if (warp < kWProd) {
    // ------------------------------------------------------------ softmax + epilogue
    // Warps 4q .. 4q + 3 own query tile q; thread t = query row t of the tile (TMEM lane t).
    reg_alloc<kTc2SoftmaxRegs>();
    const int q = warp >> 2, quarter = warp & 3;
    const int t = quarter * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t tS = tS0 + q * kTN, tO = tO0 + q * D;
    if (warp < 4) publish_block_info(p, sd, ctl.bi, bf, pr == 0 && h == 0);
    softmax_bar_sync();
    const int r = sd.q_start + (qt0 + q) * kBM + t;  // sequence-relative query row
    const bool active = q < nq;
    if (kRope && active) {
      // RoPE of this thread's query row in shared memory, before the first S product reads it
      bool okq = mbar_wait(&ctl.q_full[q], 0, wlim);
      okq = __all_sync(0xffffffffu, okq);
      if (okq && r < rows_seq)
        rope_tile_row<D>(p, sQ + q * kTileBytes, t, rope_position(p, sd, r));
      if (!okq && lane == 0) flag_timeout(p, ctl);
      fence_proxy_async_smem();  // the generic-proxy writes, before the MMAs read the tile
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.q_rot[q]);
    }
    const RowInfo ri = row_info(sd, ctl.bi, r);
    const RowMasks rm = row_masks(ri, ctl.bi, sd);
    const float sl = p.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = active;
    for (int j = 0; j < n_kt && ok; ++j) {
      const bool masked = tile_needs_mask(sd, j * kTN);
      const uint64_t vis0 = masked ? vis64(sd, j * kTN, rm) : ~0ull;
      const uint64_t vis1 = masked ? vis64(sd, j * kTN + 64, rm) : ~0ull;
      ok = !*abort_flag && mbar_wait(&ctl.s_full[q], j & 1, wlim);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      // the tile's 128 scores of this row in registers, and their maximum
      uint32_t sv[128];
      const float mt = masked ? tile_row_load<true>(tS + lane_off, vis0, vis1, sv)
                              : tile_row_load<false>(tS + lane_off, vis0, vis1, sv);
      // Raise the reference maximum on the first finite value, or when the tile maximum
      // exceeds it by more than 2^kRescaleLog2 in probability; only then is O rescaled.
      float m_new = m_run;
      if (m_run == -INFINITY) m_new = mt;
      else if ((mt - m_run) * sl > kRescaleLog2) m_new = mt;
      const bool rescale = (m_new != m_run) && (m_run != -INFINITY);
      const float alpha = rescale ? ex2_approx((m_run - m_new) * sl) : 1.f;
      const float mL = (m_new == -INFINITY) ? 0.f : m_new * sl;
      // PV_q(j - 1) completed before S_q(j) was issued: O_q may be rescaled right away.
      if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + lane_off + 32 * c, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(tO + lane_off + 32 * c, o);
        }
      }
      // P over the first 64 columns of S_q(j), and the row sum
      const uint64_t sl2 = f2_pack(sl, sl), nmL2 = f2_pack(-mL, -mL);
      uint64_t acc[4] = {0, 0, 0, 0};  // bit pattern 0 = +0.0f
      // the first half of P, handed to the PV issuer before the second is computed
      tile_row_exp<0>(tS + lane_off, sv, sl2, nmL2, acc);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.p_half[q][0]);
      tile_row_exp<1>(tS + lane_off, sv, sl2, nmL2, acc);
      float a0, a1, b0, b1;
      f2_unpack(f2_add(acc[0], acc[1]), a0, a1);
      f2_unpack(f2_add(acc[2], acc[3]), b0, b1);
      l_run = l_run * alpha + ((a0 + a1) + (b0 + b1));
      m_run = m_new;
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.p_half[q][1]);
    }
    if (active) {
      if (ok) ok = mbar_wait(&ctl.o_full[q], 0, wlim);
      const bool wok = __all_sync(0xffffffffu, ok);
      if (!wok && lane == 0) flag_timeout(p, ctl);
      // O row / row sum -> bf16 into the tile's query buffer (no MMA reads it once o_full
      // has completed), 16-byte chunks XOR-swizzled by row; then the tile's 128 threads
      // store whole rows, coalesced.
      constexpr int kChunks = D / 8;  // 16-byte chunks per output row
      uint4* stage = reinterpret_cast<uint4*>(sQ + q * kTileBytes);
      if (wok) {
        tc_fence_after();
        const float inv_l = 1.0f / l_run;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t rr[32];
          tmem_ld32(tO + lane_off + 32 * c, rr);
          tmem_wait_ld();
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            uint4 u;
            u.x = pack_bf16x2(__uint_as_float(rr[8 * v + 0]) * inv_l, __uint_as_float(rr[8 * v + 1]) * inv_l);
            u.y = pack_bf16x2(__uint_as_float(rr[8 * v + 2]) * inv_l, __uint_as_float(rr[8 * v + 3]) * inv_l);
            u.z = pack_bf16x2(__uint_as_float(rr[8 * v + 4]) * inv_l, __uint_as_float(rr[8 * v + 5]) * inv_l);
            u.w = pack_bf16x2(__uint_as_float(rr[8 * v + 6]) * inv_l, __uint_as_float(rr[8 * v + 7]) * inv_l);
            const int chunk = c * 4 + v;
            stage[t * kChunks + (chunk ^ (t & (kChunks - 1)))] = u;
          }
        }
      }
      ctl.store_row[q][t] = (wok && ri.store && r < rows_seq) ? 1 : 0;
      tile_bar_sync(q);
      if (!*abort_flag) {
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.o);
        const int rbase = row0 + sd.q_start + (qt0 + q) * kBM;
#pragma unroll 4
        for (int idx = t; idx < kBM * kChunks; idx += kBM) {
          const int row = idx / kChunks, chunk = idx % kChunks;
          if (ctl.store_row[q][row]) {
            const uint4 u = stage[row * kChunks + (chunk ^ (row & (kChunks - 1)))];
            uint4* dst = reinterpret_cast<uint4*>(
                out + (static_cast<size_t>(rbase + row) * p.hq + h) * D);
            dst[chunk] = u;
          }
        }
      }
    }
  } else {
    reg_dealloc<kTc2SideRegs>();  // warp 11: completes the side warpgroup
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kWMma) {
    // no product is still writing TMEM (both issuers committed `drained` last)
    if (lane == 0 && !mbar_wait(&ctl.drained, 0, wlim)) flag_timeout(p, ctl);
    __syncwarp();
    tc_fence_after();
    tmem_dealloc<kTmemCols>(ctl.tmem_base);
  }
}

// ---------------------------------------------------------------- host side

// Which tensor-core kernel: a cost model in SM cycles, fitted (least squares on the log of
// the time) to CUDA-graph timings of both kernels on the full and prefix-cached variants
// of four workload shapes on GB300 (within 6 % of each of the 16 timings). attn_tc1 costs
// about 14250 + 1500 kt cycles per 128-row query tile (kt = tiles of 128 keys); attn_tc2
// about 11900 + 3460 kt per pair of tiles and 32300 + 600 kt for a lone last tile (its
// chain is latency-bound, much like a pair's). Work spreads over the SMs one CTA each: a
// launch with no more CTAs than SMs takes its longest CTA, a larger one about total / SMs
// plus half a CTA of tail. attn_tc2 wins on every full workload (8B layer: one wave instead
// of 1.5, and its per-tile cost now below two of attn_tc1's), attn_tc1 on small query counts
// (the 8B prefix-cached step); where the model errs (the GQA pair) the two differ by 1.5 %.
struct TcEstimate {
  double total = 0, longest = 0;
  long long ctas = 0;
  void add(long long n, double cost) {
    if (n <= 0) return;
    total += static_cast<double>(n) * cost;
    longest = std::max(longest, cost);
    ctas += n;
  }
  double cycles(int sms) const {
    return ctas <= sms ? longest : total / sms + 0.5 * longest;
  }
};

bool prefer_tc2(const AttnParams& p, int sms) {
  TcEstimate one, two;
  for (int s = 0; s < p.num_seqs; ++s) {
    const SeqDesc& sd = p.seq[s];
    const double kt = (sd.n_orig + sd.slen + kTN - 1) / kTN;
    const long long tiles = sd.n_qtiles, heads = p.hq;
    one.add(tiles * heads, 14250.0 + 1500.0 * kt);
    two.add((tiles / 2) * heads, 11900.0 + 3460.0 * kt);
    two.add((tiles % 2) * heads, 32300.0 + 600.0 * kt);
  }
  return two.cycles(sms) < one.cycles(sms);
}


// attn_tc2's register split assumes a launch allocation of kTc2LaunchRegs per thread; with
// any other, setmaxnreg.inc would wait for registers that never come. A build that allocated
// otherwise is refused before its first launch (checked once per instantiation).
template <class F>
cudaError_t check_tc2_regs(F* kernel, std::atomic<int>& state) {
  const int known = state.load(std::memory_order_acquire);
  if (known != 0) return known == 1 ? cudaSuccess : cudaErrorInvalidDeviceFunction;
  cudaFuncAttributes fa;
  const cudaError_t e = cudaFuncGetAttributes(&fa, kernel);
  if (e != cudaSuccess) return e;
  const bool ok = fa.numRegs == static_cast<int>(kTc2LaunchRegs);
  state.store(ok ? 1 : 2, std::memory_order_release);
  return ok ? cudaSuccess : cudaErrorInvalidDeviceFunction;
}

template <int D>
cudaError_t launch_tc(const AttnParams& p, int kernel, cudaStream_t stream) {
  static std::atomic<uint64_t> attr1_done{0}, attr2_done{0}, attr2r_done{0};
  CUtensorMap mq, mk, mv;
  if (!make_map(&mk, p.k, p.hkv, D, p.total_rows, kTN) ||
      !make_map(&mv, p.v, p.hkv, D, p.total_rows, kTN))
    return cudaErrorInvalidValue;
  if (kernel == 2) {
    if (!make_map(&mq, p.q, p.hq, D, p.total_rows, kBM)) return cudaErrorInvalidValue;
    const size_t smem = tc2_smem_bytes<D>();
    static std::atomic<int> regs2{0}, regs2r{0};
    const AttnLaunch L(p.total_pairs, kTc2Threads, smem, stream, 1, p.rope != 0);
    if (p.rope) {
      cudaError_t e = check_tc2_regs(attn_tc2<D, true>, regs2r);
      if (e == cudaSuccess) e = ensure_smem_attr(attn_tc2<D, true>, smem, attr2r_done);
      return e != cudaSuccess ? e : cudaLaunchKernelEx(&L.cfg, attn_tc2<D, true>, p, mq, mk, mv);
    }
    cudaError_t e = check_tc2_regs(attn_tc2<D, false>, regs2);
    if (e == cudaSuccess) e = ensure_smem_attr(attn_tc2<D, false>, smem, attr2_done);
    return e != cudaSuccess ? e : cudaLaunchKernelEx(&L.cfg, attn_tc2<D, false>, p, mq, mk, mv);
  }
  const size_t smem = tc1_smem_bytes<D>();
  cudaError_t e = ensure_smem_attr(attn_tc1<D>, smem, attr1_done);
  if (e != cudaSuccess) return e;
  const AttnLaunch L(p.total_work, kTc1Threads, smem, stream, 1, p.rope != 0);
  return cudaLaunchKernelEx(&L.cfg, attn_tc1<D>, p, mk, mv);
}

}  // namespace

int attention_kernel_choice(const dard_attn_args& a, const AttnParams& p) {
  if (a.dtype == DARD_F32) return 3;
  // DARD_ATTN_TC=1 or 2 forces one kernel (tests and tuning); anything else: the model
  const char* force = std::getenv("DARD_ATTN_TC");
  const int forced = force ? std::atoi(force) : 0;
  if (forced == 1 || forced == 2) return forced;
  if (forced == 4) return a.head_dim == 128 ? 4 : (prefer_tc2(p, sm_count()) ? 2 : 1);
  return prefer_tc2(p, sm_count()) ? 2 : 1;
}

dard_status launch_attention(const dard_attn_args& a, AttnParams& p, cudaStream_t stream,
                             char* err, size_t err_len) {
  cudaError_t e;
  const int kernel = attention_kernel_choice(a, p);
  // Test hooks (failure-path tests; unset in normal operation): a bound on every in-kernel
  // wait, a K copy the pair kernel never issues (its waits then run out), a launch that
  // reports failure without launching.
  if (const char* w = std::getenv("DARD_TEST_WAIT_CYCLES")) p.wait_cycles = std::atoll(w);
  if (const char* d = std::getenv("DARD_TEST_DROP_KV")) p.test_drop_kv = std::atoi(d);
  if (std::getenv("DARD_TEST_FAIL_LAUNCH") != nullptr) {
    snprintf(err, err_len, "attention launch failed: %s (DARD_TEST_FAIL_LAUNCH)",
             cudaGetErrorString(cudaErrorLaunchFailure));
    return DARD_ERR_CUDA;
  }
  if (p.rope) {  // the keys are rotated once, ahead of the attention kernel
    e = launch_rope_keys(p, a.dtype, stream);
    if (e != cudaSuccess) {
      snprintf(err, err_len, "RoPE key pass launch failed: %s", cudaGetErrorString(e));
      return DARD_ERR_CUDA;
    }
  }
  if (kernel == 3) {
    e = launch_simt_attention(p, stream);
  } else if (kernel == 4) {
    e = launch_pair_attention(p, stream);
  } else {
    e = a.head_dim == 64 ? launch_tc<64>(p, kernel, stream) : launch_tc<128>(p, kernel, stream);
  }
  if (e != cudaSuccess) {
    snprintf(err, err_len, "attention launch failed: %s", cudaGetErrorString(e));
    return DARD_ERR_CUDA;
  }
  return DARD_OK;
}

}  // namespace dard
