// dard_attention_pair.cu - the state-masked attention of one DARD step on CTA pairs
// (tcgen05 cta_group::2, head_dim 128, bf16).
//
// Same arithmetic and mask as dard_attention.cu (arXiv 2608.26574 Sec. 3.1 Eq. 2; Sec. 3.2
// query blocks 1-6 and Eq. 3): every query row attends exactly one copy of every original
// position, chosen in-kernel from the block's states and c_{t-1}.
//
// Work item: 256 consecutive query rows of one (sequence, head). The two CTAs of a cluster
// (ranks 0 and 1) each hold 128 of them, and one M = 256 MMA spans both SMs: rank 0 issues
// it, A (Q, then P) and D (S, then O) are split by rows between the two CTAs' TMEM, B by
// columns between their shared memory. Each CTA therefore loads only half of every K/V
// tile: keys 64r .. 64r + 63 of K (all 128 d) and d-columns 64r .. 64r + 63 of V (all 128
// keys), 16 KB each, and feeds the tensor core half the operand bytes per MMA that a
// one-CTA kernel would.
//
// Per CTA (608 threads, one CTA per SM, persistent over work items):
//   warps 0-15 softmax and epilogue: warp w takes TMEM lane quarter w % 4 (query rows
//              32 (w % 4) .. + 31) and key columns 32 (w / 4) .. + 31 of every tile; four
//              warps share a row's maximum through shared memory. Thread 0 also loads the
//              next item's Q tile by TMA into the staging buffer;
//   warp 16    TMA producer of this CTA's K/V halves (4 stages), L2 prefetches ahead;
//   warp 17    TMEM allocation (both CTAs, collectively); rank 0 lane 0: S issuer;
//              rank 1 lane 0: forwards the landing of rank 1's K and V halves to rank 0's
//              barriers (each CTA's copies complete on its own barriers, so that every
//              CTA can wait for its own copies before it releases shared memory);
//   warp 18    rank 0 lane 0: PV issuer.
//   TMEM (each CTA): S ring [0, 256) (S(t) in buffer t % 2), O [256, 384), P [384, 448)
//   (bf16 pairs), Q [448, 512) (bf16 pairs, written by the softmax threads).
// S = Q K^T and O += P V both take A from TMEM. Two issuer threads keep the tensor pipe
// fed (its queue is short: a thread that waits on a barrier leaves it idle): S(t) needs
// only that both CTAs' softmax has read S(t - 2) out of the same buffer, PV(t) that P(t)
// is in both CTAs' TMEM; P(t + 1) replaces P(t) once PV(t) has completed. The next item's
// Q is written to TMEM as soon as the item's last S has been read, so that its first S
// products overlap this item's last PV and epilogue; its first PV waits until this item's
// O has been read out.
// The softmax keeps a per-row reference maximum and rescales O in TMEM only when the
// maximum grows by more than 2^8; the row sum adds the bf16-rounded P values that the PV
// product uses, so numerator and denominator see the same weights.
//
// Every wait is bounded. A wait that gives up sets DARD_STATUS_TIMEOUT and the abort flag;
// the softmax warps leave their loops together (their decisions are AND-reduced at named
// barriers), the producer waits (bounded) for its own copies in flight, the issuer makes
// every MMA it launched complete before TMEM is released, and both CTAs meet at a cluster
// barrier before they exit.
#include <cstdio>
#include <cstdlib>

#include "dard_attn_common.cuh"

namespace dard {
namespace {

constexpr int kSoftmaxSlots = 4;        // softmax warps per TMEM lane quarter
constexpr int kCols = kTN / kSoftmaxSlots;  // key columns of a tile per softmax thread
constexpr int kSoftmaxThreads = 128 * kSoftmaxSlots;
constexpr int kPairThreads = kSoftmaxThreads + 3 * 32;
constexpr int kPairRows = 256;          // query rows per work item (128 per CTA)
constexpr int kPD = 128;                // head_dim of this kernel
constexpr int kPST = 4;                 // K/V stages (this CTA's halves)
constexpr uint32_t kHalf = 16384;       // half of a 128-key K or V tile
constexpr uint32_t kKBlock = 8192;      // K half: two 64-key x 64-d swizzled blocks
constexpr uint16_t kBothCtas = 0x3;
constexpr int kWProducer = 4 * kSoftmaxSlots, kWIssueS = kWProducer + 1,
              kWIssuePV = kWProducer + 2;
constexpr int kSoftmaxArrivals = 2 * 4 * kSoftmaxSlots;  // softmax warps of both CTAs

struct __align__(16) PairCtl {
  uint64_t k_land[kPST], v_land[kPST];    // this CTA's half landed (TMA bytes)
  uint64_t k_peer[kPST], v_peer[kPST];    // rank 0: rank 1's half landed
  uint64_t k_empty[kPST], v_empty[kPST];  // the MMAs reading the stage completed
  uint64_t q_land;    // the next item's Q tile landed in the staging buffer (TMA bytes)
  uint64_t q_full;    // rank 0: the item's Q is in both CTAs' TMEM
  uint64_t s_full[2]; // S(t) completed in TMEM buffer t % 2
  uint64_t s_free[2]; // rank 0: both CTAs' softmax read S(t)
  uint64_t p_full;    // rank 0: P(t) is in both CTAs' TMEM
  uint64_t pv_done;   // PV(t) completed
  uint64_t o_full;    // the item's last PV completed
  uint64_t o_free;    // rank 0: both CTAs read the item's O out of TMEM
  uint64_t drained;   // every MMA both issuers launched has completed (two commits)
  uint32_t tmem_base;
  int32_t abort;
  BlockInfo bi;
  float red_max[2][kSoftmaxSlots][128];  // per tile parity: each column slot's row maxima
  float red_sum[kSoftmaxSlots][128];     // each column slot's row sums
  uint8_t store_row[128];    // epilogue: rows of this CTA that are written
};

constexpr size_t pair_smem_bytes() {
  // alignment slack + K and V stages + Q / output staging (128 rows x 256 B) + control
  return 1024 + 2 * kPST * static_cast<size_t>(kHalf) + 128 * kPD * 2 + sizeof(PairCtl);
}

// One work item: query rows [r0, r0 + 256) of (seq, head h); n_kt key tiles.
struct PairItem {
  int seq, pr, h, g, r0, n_kt;
};

__device__ __forceinline__ PairItem pair_item(const AttnParams& p, int w) {
  PairItem it;
  decode_pair(p, w, it.seq, it.pr, it.h);
  const SeqDesc& sd = p.seq[it.seq];
  it.g = it.h / (p.hq / p.hkv);
  it.r0 = sd.q_start + it.pr * kPairRows;
  const int rows = sd.n_orig + sd.slen;
  it.n_kt = key_tiles(sd, it.r0, min(it.r0 + kPairRows, rows));
  return it;
}


// N (a multiple of 32) consecutive TMEM columns of this warp's lanes, from / to registers.
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t* r) {
  static_assert(N % 32 == 0, "whole 32-column loads");
#pragma unroll
  for (int c = 0; c < N / 32; ++c)
    tmem_ld32(taddr + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(r + 32 * c));
}
template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t* r) {
  if constexpr (N == 16) {
    tmem_st16(taddr, *reinterpret_cast<const uint32_t(*)[16]>(r));
  } else {
    static_assert(N % 32 == 0, "16 or whole 32-column stores");
#pragma unroll
    for (int c = 0; c < N / 32; ++c)
      tmem_st32(taddr + 32 * c, *reinterpret_cast<const uint32_t(*)[32]>(r + 32 * c));
  }
}

// Named barrier 2 over every softmax thread of the CTA.
__device__ __forceinline__ void softmax_sync() {
  asm volatile("bar.sync 2, %0;" ::"n"(kSoftmaxThreads) : "memory");
}

__device__ __forceinline__ void pair_flag_timeout(const AttnParams& p, PairCtl& ctl) {
  ctl.abort = 1;
  if (p.status) atomicOr(p.status, DARD_STATUS_TIMEOUT);
}

__global__ void __launch_bounds__(kPairThreads, 1)
    attn_pair(const __grid_constant__ AttnParams p, const __grid_constant__ CUtensorMap tmq,
              const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv) {
  constexpr int D = kPD;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = base;                       // kPST x 16 KB
  uint8_t* sV = sK + kPST * kHalf;          // kPST x 16 KB
  uint8_t* sO = sV + kPST * kHalf;          // the next Q tile (two swizzled 16 KB blocks),
                                            // then the epilogue's 128 rows x D bf16
  PairCtl& ctl = *reinterpret_cast<PairCtl*>(sO + 128 * D * 2);

  const uint32_t rank = cluster_ctarank();  // 0 or 1 (cluster of two CTAs)
  const int cid = static_cast<int>(blockIdx.x >> 1), ncl = static_cast<int>(gridDim.x >> 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long wlim = p.wait_cycles > 0 ? p.wait_cycles : kWaitCycles;

  if (warp == kWProducer && lane == 0) {
    for (int b = 0; b < kPST; ++b) {
      mbar_init(&ctl.k_land[b], 1);
      mbar_init(&ctl.v_land[b], 1);
      mbar_init(&ctl.k_peer[b], 1);
      mbar_init(&ctl.v_peer[b], 1);
      mbar_init(&ctl.k_empty[b], 1);
      mbar_init(&ctl.v_empty[b], 1);
    }
    mbar_init(&ctl.q_land, 1);
    mbar_init(&ctl.q_full, kSoftmaxArrivals);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl.s_full[b], 1);
      mbar_init(&ctl.s_free[b], kSoftmaxArrivals);
    }
    mbar_init(&ctl.p_full, kSoftmaxArrivals);
    mbar_init(&ctl.pv_done, 1);
    mbar_init(&ctl.o_full, 1);
    mbar_init(&ctl.o_free, kSoftmaxArrivals);
    mbar_init(&ctl.drained, 2);
    ctl.abort = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmq);
    tma_prefetch_desc(&tmk);
    tma_prefetch_desc(&tmv);
  }
  if (warp == kWIssueS) {
    tmem_alloc_pair<kTmemCols>(&ctl.tmem_base);
    tmem_relinquish_pair();
  }
  // Both CTAs' barriers exist and TMEM is allocated before any CTA touches the other.
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tS = ctl.tmem_base, tO = ctl.tmem_base + 256, tP = ctl.tmem_base + 384,
                 tQ = ctl.tmem_base + 448;
  volatile int32_t* abort_flag = &ctl.abort;
  // rank 0's copy of a barrier (the one an MMA issuer waits on)
  auto lead = [](uint64_t* bar) { return map_shared_rank(smem_u32(bar), 0); };

  if (warp == kWProducer) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int use = 0;
      int k_last[kPST], v_last[kPST];  // the latest use of each stage whose copy was issued
      for (int b = 0; b < kPST; ++b) k_last[b] = v_last[b] = -1;
      bool ok = true;
      grid_dep_wait();  // the RoPE key pass launched before this kernel (if any) is complete
      for (int w = cid; w < p.total_pairs && ok; w += ncl) {
        const PairItem it = pair_item(p, w);
        const int row0 = p.seq[it.seq].row_base;
        const int kc = it.g * D;  // first column of the K/V head
        auto prefetch = [&](int j) {
          tma_prefetch_l2_2d(&tmk, kc, row0 + j * kTN + 64 * rank);
          tma_prefetch_l2_2d(&tmk, kc + 64, row0 + j * kTN + 64 * rank);
          tma_prefetch_l2_2d(&tmv, kc + 64 * rank, row0 + j * kTN);
        };
        for (int j = 0; j < kL2Ahead && j < it.n_kt; ++j) prefetch(j);
        for (int j = 0; j < it.n_kt; ++j, ++use) {
          if (j + kL2Ahead < it.n_kt) prefetch(j + kL2Ahead);
          const int b = use % kPST;
          const uint32_t ph = ((use / kPST) - 1) & 1;
          ok = !*abort_flag && (use < kPST || mbar_wait(&ctl.k_empty[b], ph, wlim));
          if (!ok) break;
          mbar_arrive_expect_tx(&ctl.k_land[b], kHalf);
          if (use != p.test_drop_kv) {  // test hook: a dropped copy is never issued
            tma_load_2d(sK + b * kHalf, &tmk, &ctl.k_land[b], kc, row0 + j * kTN + 64 * rank);
            tma_load_2d(sK + b * kHalf + kKBlock, &tmk, &ctl.k_land[b], kc + 64,
                        row0 + j * kTN + 64 * rank);
            k_last[b] = use;
          }
          ok = use < kPST || mbar_wait(&ctl.v_empty[b], ph, wlim);
          if (!ok) break;
          mbar_arrive_expect_tx(&ctl.v_land[b], kHalf);
          tma_load_2d(sV + b * kHalf, &tmv, &ctl.v_land[b], kc + 64 * rank, row0 + j * kTN);
          v_last[b] = use;
        }
      }
      if (!ok) pair_flag_timeout(p, ctl);
      // Every copy this CTA issued lands before shared memory is released: the latest
      // issued use of each stage (earlier uses of a stage landed before it was reused).
      for (int b = 0; b < kPST; ++b) {
        if (k_last[b] >= 0 && !mbar_wait(&ctl.k_land[b], (k_last[b] / kPST) & 1, wlim))
          pair_flag_timeout(p, ctl);
        if (v_last[b] >= 0 && !mbar_wait(&ctl.v_land[b], (v_last[b] / kPST) & 1, wlim))
          pair_flag_timeout(p, ctl);
      }
    }
  } else if (warp == kWIssueS) {
    if (rank == 0 && lane == 0) {
      // ---------------------------------------------------------- S issuer (rank 0)
      // S(t) = Q K(t)^T into buffer t % 2, once K(t) has landed in both CTAs and both
      // CTAs' softmax has read S(t - 2) out of the buffer; the item's first S once its Q
      // is in both CTAs' TMEM.
      constexpr uint32_t kIdS = idesc_bf16_f32(2 * kBM, kTN, 0, 0);
      const uint32_t ak = smem_u32(sK);
      int s_it = 0, item_it = 0;
      bool ok = true;
      for (int w = cid; w < p.total_pairs && ok; w += ncl, ++item_it) {
        const PairItem it = pair_item(p, w);
        ok = !*abort_flag && mbar_wait(&ctl.q_full, item_it & 1, wlim);
        for (int j = 0; j < it.n_kt && ok; ++j, ++s_it) {
          const int b = s_it & 1, kb = s_it % kPST;
          const uint32_t kph = (s_it / kPST) & 1;
          ok = (s_it < 2 || mbar_wait(&ctl.s_free[b], ((s_it >> 1) - 1) & 1, wlim)) &&
               mbar_wait(&ctl.k_land[kb], kph, wlim) && mbar_wait(&ctl.k_peer[kb], kph, wlim);
          if (!ok) break;
          tc_fence_after();
          const uint32_t kaddr = ak + kb * kHalf;
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks)
            mma_ts_pair(tS + b * kTN, tQ + ks * 8,
                        smem_desc_sw128(kaddr + (ks >> 2) * kKBlock + (ks & 3) * 32, 16, 1024),
                        kIdS, ks > 0);
          mma_commit_pair(&ctl.s_full[b], kBothCtas);
          mma_commit_pair(&ctl.k_empty[kb], kBothCtas);
        }
        if (*abort_flag) ok = false;
      }
      if (!ok) pair_flag_timeout(p, ctl);
      mma_commit_pair(&ctl.drained, kBothCtas);  // completes once every S MMA has
    } else if (rank == 1 && lane == 0) {
      // ---------------------------------------------------------- landing forwarder
      // K then V of every use, in the producer's order (one thread: a waiting lane would
      // hold up any other lane of its warp).
      int use = 0;
      bool ok = true;
      for (int w = cid; w < p.total_pairs && ok; w += ncl) {
        const PairItem it = pair_item(p, w);
        for (int j = 0; j < it.n_kt; ++j, ++use) {
          const int b = use % kPST;
          const uint32_t ph = (use / kPST) & 1;
          ok = !*abort_flag && mbar_wait(&ctl.k_land[b], ph, wlim);
          if (!ok) break;
          mbar_arrive_remote(lead(&ctl.k_peer[b]));
          ok = mbar_wait(&ctl.v_land[b], ph, wlim);
          if (!ok) break;
          mbar_arrive_remote(lead(&ctl.v_peer[b]));
        }
      }
      if (!ok) pair_flag_timeout(p, ctl);
    }
  } else if (warp == kWIssuePV) {
    if (rank == 0 && lane == 0) {
      // ---------------------------------------------------------- PV issuer (rank 0)
      // O (+)= P(t) V(t), once P(t) is in both CTAs' TMEM and V(t) has landed in both; the
      // item's first PV (which overwrites O) once the previous item's O has been read out.
      constexpr uint32_t kIdO = idesc_bf16_f32(2 * kBM, D, 0, 1);
      const uint32_t av = smem_u32(sV);
      int pv_it = 0, item_it = 0;
      bool ok = true;
      for (int w = cid; w < p.total_pairs && ok; w += ncl, ++item_it) {
        const PairItem it = pair_item(p, w);
        for (int j = 0; j < it.n_kt && ok; ++j, ++pv_it) {
          const int vb = pv_it % kPST;
          const uint32_t vph = (pv_it / kPST) & 1;
          ok = !*abort_flag && mbar_wait(&ctl.p_full, pv_it & 1, wlim) &&
               (j > 0 || item_it == 0 || mbar_wait(&ctl.o_free, (item_it - 1) & 1, wlim)) &&
               mbar_wait(&ctl.v_land[vb], vph, wlim) && mbar_wait(&ctl.v_peer[vb], vph, wlim);
          if (!ok) break;
          tc_fence_after();
          const uint32_t vaddr = av + vb * kHalf;
#pragma unroll
          for (int ks = 0; ks < kTN / 16; ++ks)
            mma_ts_pair(tO, tP + ks * 8, smem_desc_sw128(vaddr + ks * 2048, kHalf, 1024), kIdO,
                        (j > 0 || ks > 0) ? 1u : 0u);
          mma_commit_pair(&ctl.pv_done, kBothCtas);
          mma_commit_pair(&ctl.v_empty[vb], kBothCtas);
          if (j == it.n_kt - 1) mma_commit_pair(&ctl.o_full, kBothCtas);
        }
      }
      if (!ok) pair_flag_timeout(p, ctl);
      mma_commit_pair(&ctl.drained, kBothCtas);  // completes once every PV MMA has
    }
  } else {
    // ------------------------------------------------------------ softmax + epilogue
    // Warp w: TMEM lane quarter w % 4 (query rows 32 (w % 4) .. + 31), column slot w / 4
    // (keys 32 slot .. + 31 of a tile, P columns 16 slot .., O and Q columns 32 slot ..).
    const int quarter = warp & 3, slot = warp >> 2;
    const int t = quarter * 32 + lane;  // TMEM lane = this CTA's query row within the item
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const float sl = p.scale_log2;
    BlockFetch bf{-1, 0.f, -1};
    // Thread 0: the Q tile of an item (this CTA's 128 rows, two 64-column swizzled blocks)
    // by TMA into the staging buffer, which is free (every softmax thread has passed the
    // barrier after its last use).
    int q_loads = 0;   // Q tiles taken out of the staging buffer so far (q_land phases)
    int q_issued = 0;  // Q tile loads issued (thread 0)
    auto load_q = [&](const PairItem& qi) {
      if (threadIdx.x == 0) {
        ++q_issued;
        const int row = p.seq[qi.seq].row_base + qi.r0 + kBM * static_cast<int>(rank);
        fence_proxy_async_smem();  // the buffer's generic reads and writes come first
        mbar_arrive_expect_tx(&ctl.q_land, 2 * kHalf);
        tma_load_2d(sO, &tmq, &ctl.q_land, qi.h * D, row);
        tma_load_2d(sO + kHalf, &tmq, &ctl.q_land, qi.h * D + 64, row);
      }
    };
    // This thread's kCols elements of its query row in item qi (d = kCols slot .., 16-byte
    // chunks of row t in the staging buffer), with RoPE when asked for, into TMEM (bf16
    // pairs), then tell rank 0.
    auto store_q = [&](const PairItem& qi) -> bool {
      bool okq = mbar_wait(&ctl.q_land, q_loads & 1, wlim);
      okq = __all_sync(0xffffffffu, okq);
      ++q_loads;
      if (!okq) return false;
      const SeqDesc& qsd = p.seq[qi.seq];
      const int qr = qi.r0 + kBM * static_cast<int>(rank) + t;  // sequence-relative row
      const bool rot = p.rope && qr < qsd.n_orig + qsd.slen;
      const int pos = rot ? rope_position(p, qsd, qr) : 0;
      uint32_t qw[kCols / 2];
#pragma unroll
      for (int c = 0; c < kCols / 8; ++c) {
        const int cg = (kCols / 8) * slot + c;  // chunk of the row: elements 8 cg .. 8 cg + 7
        uint4 u = *sw128_chunk(sO, t, cg);
        if (rot) {
          if (p.rope_style == DARD_ROPE_INTERLEAVED)
            rope_chunk_interleaved(u, pos, p.rope_f + 8 * cg);
          else  // the partner chunk D/2 elements away, in the other 64-column block
            rope_chunk_half(u, *sw128_chunk(sO, t, cg ^ 8), cg < 8, pos, p.rope_f + 16 * (cg & 7));
        }
        qw[4 * c + 0] = u.x;
        qw[4 * c + 1] = u.y;
        qw[4 * c + 2] = u.z;
        qw[4 * c + 3] = u.w;
      }
      tmem_st_cols<kCols / 2>(tQ + lane_off + slot * (kCols / 2), qw);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(lead(&ctl.q_full));
      return true;
    };
    int w = cid, tg = 0, item_it = 0;
    PairItem it{};
    bool run = w < p.total_pairs;
    if (run) {
      it = pair_item(p, w);
      load_q(it);
      if (warp < 4) bf = fetch_block_info(p, p.seq[it.seq]);
      run = store_q(it);
    }
    run = bar_and(2, kSoftmaxThreads, run);  // and every thread has read the staging buffer
    if (run && w + ncl < p.total_pairs) load_q(pair_item(p, w + ncl));
    for (; run && w < p.total_pairs; w += ncl, ++item_it) {
      const SeqDesc sd = p.seq[it.seq];  // a register copy: the loop reads it every tile
      const int rows_seq = sd.n_orig + sd.slen;
      const int rs = it.r0 + kBM * static_cast<int>(rank) + t;  // sequence-relative row
      // The block of this item's sequence (every softmax warp is done with the previous
      // item's copy: it passed that item's epilogue barriers).
      if (warp < 4) publish_block_info(p, sd, ctl.bi, bf, it.pr == 0 && it.h == 0 && rank == 0);
      softmax_sync();
      bool store_row;  // this thread's row is an output row of the call
      RowMasks rm;
      {
        const RowInfo ri = row_info(sd, ctl.bi, rs);
        rm = row_masks(ri, ctl.bi, sd);
        store_row = ri.store && rs < rows_seq;
      }
      // the next item's block (its Q tile is on its way already)
      const bool has_next = w + ncl < p.total_pairs;
      if (has_next && warp < 4) bf = fetch_block_info(p, p.seq[pair_item(p, w + ncl).seq]);
      float m_run = -INFINITY, l_run = 0.f;
      bool ok = true;
      for (int j = 0; j < it.n_kt; ++j, ++tg) {
        const int b = tg & 1;
        const bool masked = tile_needs_mask(sd, j * kTN);
        // visibility of this thread's kCols keys (64 per word)
        uint64_t vis[(kCols + 63) / 64];
#pragma unroll
        for (int c = 0; c < (kCols + 63) / 64; ++c)
          vis[c] = masked ? vis64(sd, j * kTN + kCols * slot + 64 * c, rm) : ~0ull;
        bool wok = ok && !*abort_flag && mbar_wait(&ctl.s_full[b], (tg >> 1) & 1, wlim);
        wok = __all_sync(0xffffffffu, wok);
        float s[kCols];
        float mh = -INFINITY;
        if (wok) {
          tc_fence_after();
          uint32_t r[kCols];
          tmem_ld_cols<kCols>(tS + b * kTN + kCols * slot + lane_off, r);
          tmem_wait_ld();
          // S(t) is in registers: rank 0 may reuse its buffer for S(t + 2)
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_remote(lead(&ctl.s_free[b]));
#pragma unroll
          for (int e = 0; e < kCols; ++e) s[e] = __uint_as_float(r[e]);
          if (masked) {
#pragma unroll
            for (int k = 0; k < kCols; ++k)
              s[k] = ((vis[k / 64] >> (k % 64)) & 1ull) ? s[k] : -INFINITY;
          }
          float mx[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) mx[e] = s[e];
#pragma unroll
          for (int k = 8; k < kCols; k += 8) {
#pragma unroll
            for (int e = 0; e < 8; ++e) mx[e] = fmaxf(mx[e], s[k + e]);
          }
          mh = fmaxf(fmax3(mx[0], mx[1], mx[2]), fmax3(fmax3(mx[3], mx[4], mx[5]), mx[6], mx[7]));
          if (kSoftmaxSlots > 1) ctl.red_max[tg & 1][slot][t] = mh;
        }
        // the warps of the rows leave together, or all go on with all their maxima
        if (!bar_and(3 + quarter, 32 * kSoftmaxSlots, wok)) {
          ok = false;
          break;
        }
        float mt = mh;
        if (kSoftmaxSlots > 1) {
          mt = ctl.red_max[tg & 1][0][t];
#pragma unroll
          for (int sl2 = 1; sl2 < kSoftmaxSlots; ++sl2) mt = fmaxf(mt, ctl.red_max[tg & 1][sl2][t]);
        }
        // Raise the reference maximum on the first finite value, or when the tile maximum
        // exceeds it by more than 2^kRescaleLog2 in probability; only then is O rescaled.
        // The warps of a row take the same decision from the same values.
        float m_new = m_run;
        if (m_run == -INFINITY) m_new = mt;
        else if ((mt - m_run) * sl > kRescaleLog2) m_new = mt;
        const bool rescale = (m_new != m_run) && (m_run != -INFINITY);
        const float alpha = rescale ? ex2_approx((m_run - m_new) * sl) : 1.f;
        const float mL = (m_new == -INFINITY) ? 0.f : m_new * sl;
        uint32_t pk[kCols / 2];
        const uint64_t sl2 = f2_pack(sl, sl), nmL2 = f2_pack(-mL, -mL);
        uint64_t acc[2] = {0, 0};  // two packed partial sums (bit pattern 0 = +0.0f)
#pragma unroll
        for (int e = 0; e < kCols / 2; ++e) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(s[2 * e], s[2 * e + 1]), sl2, nmL2), x0, x1);
          pk[e] = pack_bf16x2(ex2_approx(x0), ex2_approx(x1));
          // the row sum adds the rounded weights the PV product multiplies with
          acc[e & 1] = f2_add(acc[e & 1], f2_pack(__uint_as_float(pk[e] << 16),
                                                  __uint_as_float(pk[e] & 0xffff0000u)));
        }
        float a0, a1;
        f2_unpack(f2_add(acc[0], acc[1]), a0, a1);
        // P(t) replaces P(t - 1), and O may be rescaled, once PV(t - 1) has completed
        wok = tg == 0 || mbar_wait(&ctl.pv_done, (tg - 1) & 1, wlim);
        wok = __all_sync(0xffffffffu, wok);
        if (!wok) {
          // leave with the other warps of the rows at the next tile's barrier (or the
          // epilogue's)
          ok = false;
          continue;
        }
        tc_fence_after();
        tmem_st_cols<kCols / 2>(tP + lane_off + (kCols / 2) * slot, pk);
        // O (stable: PV(t - 1) completed, PV(t) waits for the arrival below) is rescaled
        // only when the reference maximum moved
        if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll 1
          for (int c = 0; c < kCols / 16; ++c) {  // this warp's kCols O columns
            uint32_t r[16];
            const uint32_t col = tO + lane_off + kCols * slot + 16 * c;
            tmem_ld16(col, r);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
            tmem_st16(col, r);
          }
        }
        l_run = l_run * alpha + (a0 + a1);
        m_run = m_new;
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(lead(&ctl.p_full));
      }
      // The item's last S has been read: the next item's Q may replace this one in TMEM,
      // so that its first S products run during this item's last PV and epilogue.
      bool go_on = ok && has_next;
      if (go_on) go_on = store_q(pair_item(p, w + ncl));
      // ---------------------------------------------------------- epilogue
      bool wok = ok && mbar_wait(&ctl.o_full, item_it & 1, wlim);
      wok = __all_sync(0xffffffffu, wok);
      ctl.red_sum[slot][t] = l_run;
      const bool all_ok = bar_and(2, kSoftmaxThreads, wok);  // every warp's verdict, and sync
      if (!all_ok && lane == 0 && !wok) pair_flag_timeout(p, ctl);
      constexpr int kChunks = D / 8;  // 16-byte chunks per output row
      uint4* stage = reinterpret_cast<uint4*>(sO);
      if (all_ok) {
        tc_fence_after();
        float lsum = ctl.red_sum[0][t];
#pragma unroll
        for (int sl2 = 1; sl2 < kSoftmaxSlots; ++sl2) lsum += ctl.red_sum[sl2][t];
        const float inv_l = 1.0f / lsum;
#pragma unroll
        for (int c = 0; c < kCols / 32; ++c) {  // this warp's kCols O columns, 32 at a time
          uint32_t rr[32];
          tmem_ld32(tO + lane_off + kCols * slot + 32 * c, rr);
          tmem_wait_ld();
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            uint4 u;
            u.x = pack_bf16x2(__uint_as_float(rr[8 * v + 0]) * inv_l, __uint_as_float(rr[8 * v + 1]) * inv_l);
            u.y = pack_bf16x2(__uint_as_float(rr[8 * v + 2]) * inv_l, __uint_as_float(rr[8 * v + 3]) * inv_l);
            u.z = pack_bf16x2(__uint_as_float(rr[8 * v + 4]) * inv_l, __uint_as_float(rr[8 * v + 5]) * inv_l);
            u.w = pack_bf16x2(__uint_as_float(rr[8 * v + 6]) * inv_l, __uint_as_float(rr[8 * v + 7]) * inv_l);
            const int chunk = slot * (kCols / 8) + 4 * c + v;
            stage[t * kChunks + (chunk ^ (t & (kChunks - 1)))] = u;
          }
        }
        // O has been read out: rank 0 may start the next item's first PV
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(lead(&ctl.o_free));
      }
      if (slot == 0) ctl.store_row[t] = (all_ok && store_row) ? 1 : 0;
      softmax_sync();
      if (all_ok) {
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.o);
        const size_t rbase = static_cast<size_t>(sd.row_base) + it.r0 + kBM * rank;
#pragma unroll 4
        for (int idx = threadIdx.x; idx < kBM * kChunks; idx += kSoftmaxThreads) {
          const int row = idx / kChunks, chunk = idx % kChunks;
          if (ctl.store_row[row]) {
            const uint4 u = stage[row * kChunks + (chunk ^ (row & (kChunks - 1)))];
            uint4* dst = reinterpret_cast<uint4*>(out + ((rbase + row) * p.hq + it.h) * D);
            dst[chunk] = u;
          }
        }
      }
      // the staging buffer takes the next Q tile only after every thread has stored from it
      const bool cont = bar_and(2, kSoftmaxThreads, all_ok && go_on);
      if (!cont) break;
      if (w + 2 * ncl < p.total_pairs) load_q(pair_item(p, w + 2 * ncl));
      it = pair_item(p, w + ncl);
    }
    // A Q tile load issued but not taken out (an item left early) lands before shared
    // memory is released; at most the latest one is outstanding.
    if (threadIdx.x == 0 && q_issued > q_loads &&
        !mbar_wait(&ctl.q_land, (q_issued - 1) & 1, wlim))
      pair_flag_timeout(p, ctl);
  }
  // ------------------------------------------------------------ teardown
  __syncwarp();
  tc_fence_before();
  cluster_sync();  // no CTA leaves while the other may still signal its barriers
  if (warp == kWIssueS) {
    // every MMA rank 0 issued has completed (each issuer committed `drained` after its
    // last one)
    if (!mbar_wait(&ctl.drained, 0, wlim) && lane == 0) pair_flag_timeout(p, ctl);
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair<kTmemCols>(ctl.tmem_base);
  }
}

// Clusters of this kernel that fit on the device at once (one CTA per SM), per device.
int pair_max_clusters(size_t smem) {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  int n = cache[dev].load(std::memory_order_relaxed);
  if (n > 0) return n;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * 64);
  cfg.blockDim = dim3(kPairThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaOccupancyMaxActiveClusters(&n, attn_pair, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return sm_count() / 2;  // not cached: the query may succeed once the attributes are set
  }
  cache[dev].store(n, std::memory_order_relaxed);
  return n;
}

}  // namespace

int pair_clusters_for(const AttnParams& p) {
  return std::max(1, std::min(p.total_pairs, pair_max_clusters(pair_smem_bytes())));
}

cudaError_t launch_pair_attention(const AttnParams& p, cudaStream_t stream) {
  static std::atomic<uint64_t> attr_done{0};
  CUtensorMap mq, mk, mv;
  if (!make_map(&mq, p.q, p.hq, kPD, p.total_rows, kBM) ||
      !make_map(&mk, p.k, p.hkv, kPD, p.total_rows, 64) ||
      !make_map(&mv, p.v, p.hkv, kPD, p.total_rows, kTN))
    return cudaErrorInvalidValue;
  const size_t smem = pair_smem_bytes();
  cudaError_t e = ensure_smem_attr(attn_pair, smem, attr_done);
  if (e != cudaSuccess) return e;
  const AttnLaunch L(2 * pair_clusters_for(p), kPairThreads, smem, stream, 2, p.rope != 0);
  return cudaLaunchKernelEx(&L.cfg, attn_pair, p, mq, mk, mv);
}

}  // namespace dard
