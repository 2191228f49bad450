// dard_attn_common.cuh - pieces shared by the attention kernels (dard_attention.cu,
// dard_attention_pair.cu): the per-CTA copy of the current block, the in-kernel mask of
// Sec. 3.2 (which copy, x^j or s^j, a query attends for every position j), the ragged
// work decoding, and the host helpers for tensor maps and kernel attributes.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <climits>
#include <cmath>
#include <mutex>

#include "dard_internal.h"
#include "dard_ptx.cuh"
#include "dard_rope.cuh"

namespace dard {
namespace {


constexpr int kBM = 128;  // query rows per CTA
constexpr uint32_t kTmemCols = 512;  // every TMEM column of the SM
constexpr float kRescaleLog2 = 8.0f;

// Per-CTA copy of the current block: states, confidences, the shadow maps, and the same
// facts as bit words over block positions (word w = positions 32w .. 32w + 31).
struct __align__(16) BlockInfo {
  int32_t st[DARD_MAX_BLOCK];
  float cf[DARD_MAX_BLOCK];
  int32_t shrow[DARD_MAX_BLOCK];  // block position -> shadow row index k, or -1
  int32_t shpos[DARD_MAX_BLOCK];  // shadow row index k -> block position, or -1 if invalid
  uint32_t m_w[4], c_w[4], hs_w[4];  // state M, state C, has a (valid) shadow row
  int32_t identity;                  // shpos[k] == k for every shadow row
};

// The query a row stands for: its copy (x or s), its state, c_{t-1}, block position.
struct RowInfo {
  int qs;     // 1 for a shadow query s^i
  int si;     // state of position i
  float ci;   // c_{t-1} of position i (block positions only)
  int i;      // block position of i, or -1 outside the block
  int store;  // 0 for padding rows and invalid shadow rows
};

__device__ __forceinline__ void sm_bar_sync() {  // warps 0-3 only
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

__device__ __forceinline__ void decode_work(const AttnParams& p, int w, int& seq, int& qt,
                                            int& h) {
  int lo = 0, hi = p.num_seqs;  // work_prefix[lo] <= w < work_prefix[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.work_prefix[mid] <= w) lo = mid; else hi = mid;
  }
  seq = p.order[lo];
  const int local = w - p.work_prefix[lo];
  h = local % p.hq;
  qt = local / p.hq;
}

// The same over pairs of query tiles (the tensor-core path): work item w is query-tile pair
// pr of head h of sequence seq.
__device__ __forceinline__ void decode_pair(const AttnParams& p, int w, int& seq, int& pr,
                                            int& h) {
  int lo = 0, hi = p.num_seqs;  // pair_prefix[lo] <= w < pair_prefix[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.pair_prefix[mid] <= w) lo = mid; else hi = mid;
  }
  seq = p.order[lo];
  const int local = w - p.pair_prefix[lo];
  h = local % p.hq;
  pr = local / p.hq;
}

// The block's per-position data as one thread fetches it from global memory (thread t:
// block position t and shadow row t), so that the loads can be in flight early.
struct BlockFetch {
  int st;    // state of block position t, or -1
  float cf;  // c_{t-1} of block position t
  int pos;   // block position of shadow row t, or -1 past S
};

__device__ __forceinline__ BlockFetch fetch_block_info(const AttnParams& p, const SeqDesc& sd) {
  const int t = threadIdx.x;
  BlockFetch f{-1, 0.f, -1};
  if (t < sd.blen) {
    f.st = p.state[sd.blk_off + t];
    f.cf = p.prev_conf[sd.blk_off + t];
  }
  if (t < sd.slen) f.pos = p.shadow_src[sd.sh_off + t] - sd.b0;
  return f;
}

// Called by the 128 threads of warps 0-3. A repeated shadow position keeps its lowest
// shadow row; the others, and positions outside the block, are flagged and never used.
__device__ void publish_block_info(const AttnParams& p, const SeqDesc& sd, BlockInfo& bi,
                                   const BlockFetch& f, bool report) {
  const int t = threadIdx.x;
  bi.shrow[t] = INT_MAX;
  bi.shpos[t] = -1;
  if (t < sd.blen) {
    int s = f.st;
    if (s > 2) {
      if (report && p.status) atomicOr(p.status, DARD_STATUS_BAD_STATE);
      s = kStateM;
    }
    bi.st[t] = s;
    bi.cf[t] = f.cf;
  }
  const int pos = f.pos;
  const bool in_block = t < sd.slen && pos >= 0 && pos < sd.blen;
  sm_bar_sync();
  if (in_block) atomicMin(&bi.shrow[pos], t);
  sm_bar_sync();
  if (t < sd.slen) {
    const bool ok = in_block && bi.shrow[pos] == t;
    if (ok) bi.shpos[t] = pos;
    else if (report && p.status) atomicOr(p.status, DARD_STATUS_BAD_SHADOW);
  }
  sm_bar_sync();
  if (bi.shrow[t] == INT_MAX) bi.shrow[t] = -1;
  const int lane = t & 31, w = t >> 5;
  const int s_t = t < sd.blen ? bi.st[t] : -1;
  const uint32_t mw = __ballot_sync(0xffffffffu, s_t == kStateM);
  const uint32_t cw = __ballot_sync(0xffffffffu, s_t == kStateC);
  const uint32_t hw = __ballot_sync(0xffffffffu, t < sd.blen && bi.shrow[t] >= 0);
  const uint32_t idw = __ballot_sync(0xffffffffu, t >= sd.slen || bi.shpos[t] == t);
  if (lane == 0) {
    bi.m_w[w] = mw;
    bi.c_w[w] = cw;
    bi.hs_w[w] = hw;
  }
  if (t == 0) bi.identity = 1;
  sm_bar_sync();
  if (lane == 0 && idw != 0xffffffffu) bi.identity = 0;
  sm_bar_sync();
}

__device__ __forceinline__ void load_block_info(const AttnParams& p, const SeqDesc& sd,
                                                BlockInfo& bi, bool report) {
  publish_block_info(p, sd, bi, fetch_block_info(p, sd), report);
}

__device__ __forceinline__ RowInfo row_info(const SeqDesc& sd, const BlockInfo& bi, int r) {
  RowInfo q{0, kStateU, 0.f, -1, 1};
  if (r < sd.n_orig) {
    const int j = r - sd.b0;
    if (j >= 0 && j < sd.blen) {
      q.i = j;
      q.si = bi.st[j];
      q.ci = bi.cf[j];
    } else {
      q.si = (r < sd.b0) ? kStateU : kStateM;  // decoded context / future blocks
    }
  } else if (r < sd.n_orig + sd.slen) {
    const int j = bi.shpos[r - sd.n_orig];
    q.qs = 1;
    if (j >= 0) {
      q.i = j;
      q.si = bi.st[j];
      q.ci = bi.cf[j];
    } else {
      q.store = 0;
    }
  } else {
    q.store = 0;
  }
  return q;
}

// Sec. 3.2: does query q take the shadow copy s^j (true) or x^j (false) of block position j?
__device__ __forceinline__ bool takes_shadow(const RowInfo& q, int sj, float cj, int j) {
  if (sj == kStateU) return q.qs && j == q.i;           // blocks 3/6: only the own position
  if (sj == kStateM) return q.qs || q.si != kStateM;    // block 1 keeps x, all others s
  if (q.si == kStateM) return q.qs;                     // block 1: x, block 4: s
  if (q.si == kStateU) return true;                     // blocks 3/6: C keys from s
  return !(q.ci <= cj) || (q.qs && j == q.i);           // blocks 2/5: Eq. 3
}

// Whether key row kr (sequence-relative) is attended by query q.
__device__ __forceinline__ bool key_visible(const RowInfo& q, const BlockInfo& bi,
                                            const SeqDesc& sd, int kr) {
  if (kr >= sd.n_orig + sd.slen) return false;
  if (kr >= sd.n_orig) {
    const int j = bi.shpos[kr - sd.n_orig];
    return j >= 0 && takes_shadow(q, bi.st[j], bi.cf[j], j);
  }
  const int j = kr - sd.b0;
  if (j >= 0 && j < sd.blen) return !(bi.shrow[j] >= 0 && takes_shadow(q, bi.st[j], bi.cf[j], j));
  return true;
}

// ---------------------------------------------------------------- tensor-core path
// Row masks over block positions (bit j = block position j), or over shadow rows.
struct Bits128 {
  uint64_t lo, hi;
};

__device__ __forceinline__ void set_bit(Bits128& b, int j) {
  if (j < 64) b.lo |= 1ull << j; else b.hi |= 1ull << (j - 64);
}
__device__ __forceinline__ bool get_bit(const Bits128& b, int j) {
  return ((j < 64 ? b.lo >> j : b.hi >> (j - 64)) & 1ull) != 0;
}
// 64 bits of b starting at bit `start` (0 <= start); bits past 127 read as 0.
__device__ __forceinline__ uint64_t bits_window(const Bits128& b, int start) {
  if (start >= 128) return 0;
  if (start >= 64) return b.hi >> (start - 64);
  if (start == 0) return b.lo;
  return (b.lo >> start) | (b.hi << (64 - start));
}

// Per query row, the two masks the tiles need: block positions whose x copy the row does
// not see (it takes the shadow copy and the position has one), and shadow rows it sees.
struct RowMasks {
  Bits128 hide_x;
  Bits128 see_s;
};

__device__ __forceinline__ Bits128 words128(const uint32_t (&w)[4]) {
  return {static_cast<uint64_t>(w[0]) | (static_cast<uint64_t>(w[1]) << 32),
          static_cast<uint64_t>(w[2]) | (static_cast<uint64_t>(w[3]) << 32)};
}
__device__ __forceinline__ Bits128 low_bits(int n) {  // bits [0, n), 0 <= n <= 128
  Bits128 b;
  b.lo = n >= 64 ? ~0ull : ((1ull << n) - 1);
  b.hi = n >= 128 ? ~0ull : (n > 64 ? ((1ull << (n - 64)) - 1) : 0ull);
  return b;
}

// The rule of takes_shadow() over all block positions at once, from the class words.
__device__ RowMasks row_masks(const RowInfo& q, const BlockInfo& bi, const SeqDesc& sd) {
  const Bits128 mb = words128(bi.m_w), cb = words128(bi.c_w), hs = words128(bi.hs_w);
  Bits128 ts{0, 0};
  if (q.si == kStateU || (q.si == kStateM && q.qs)) {
    ts = {mb.lo | cb.lo, mb.hi | cb.hi};
  } else if (q.si == kStateC) {
    // C keys with !(c_i <= c_j) come from s (Eq. 3); confidences read four at a time
    Bits128 lower{0, 0};
    const float4* cf4 = reinterpret_cast<const float4*>(bi.cf);
    for (int j4 = 0; j4 < (sd.blen + 3) / 4; ++j4) {
      const float4 c = cf4[j4];
      const uint64_t nib = static_cast<uint64_t>(!(q.ci <= c.x)) |
                           (static_cast<uint64_t>(!(q.ci <= c.y)) << 1) |
                           (static_cast<uint64_t>(!(q.ci <= c.z)) << 2) |
                           (static_cast<uint64_t>(!(q.ci <= c.w)) << 3);
      const int j = 4 * j4;
      if (j < 64) lower.lo |= nib << j; else lower.hi |= nib << (j - 64);
    }
    ts = {mb.lo | (cb.lo & lower.lo), mb.hi | (cb.hi & lower.hi)};
  }
  if (q.qs && q.i >= 0) set_bit(ts, q.i);  // a shadow query takes its own shadow key
  RowMasks m;
  m.hide_x = {ts.lo & hs.lo, ts.hi & hs.hi};
  if (bi.identity) {
    const Bits128 lim = low_bits(sd.slen);
    m.see_s = {ts.lo & lim.lo, ts.hi & lim.hi};
  } else {
    m.see_s = {0, 0};
    const int4* sp4 = reinterpret_cast<const int4*>(bi.shpos);
    for (int k4 = 0; k4 < (sd.slen + 3) / 4; ++k4) {
      const int4 jj = sp4[k4];
      const int js[4] = {jj.x, jj.y, jj.z, jj.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int k = 4 * k4 + e;
        if (k < sd.slen && js[e] >= 0 && get_bit(ts, js[e])) set_bit(m.see_s, k);
      }
    }
  }
  return m;
}

constexpr int kTN = 128;  // keys per tile of the tensor-core path
constexpr int kL2Ahead = 4;  // K/V tiles the CTA-pair kernel prefetches into L2 ahead of its
                              // TMA loads (the one- and two-tile kernels: none, measured faster)

static_assert(kTN == kKeyTile, "one key-tile width for the kernels and the planner");

__device__ __forceinline__ bool tile_needs_mask(const SeqDesc& sd, int kt0) {
  return (kt0 + kTN > sd.n_orig) ||
         (sd.blen > 0 && kt0 < sd.b0 + sd.blen && kt0 + kTN > sd.b0);
}

// Visibility of keys [kt0, kt0 + 64) for one row (bit t = key kt0 + t).
__device__ __forceinline__ uint64_t vis64(const SeqDesc& sd, int kt0, const RowMasks& m) {
  uint64_t vis = ~0ull;
  const int lo = max(kt0, sd.b0), hi = min(kt0 + 64, sd.b0 + sd.blen);
  if (lo < hi) {
    const int len = hi - lo;
    uint64_t h = bits_window(m.hide_x, lo - sd.b0);
    if (len < 64) h &= (1ull << len) - 1;
    vis &= ~(h << (lo - kt0));
  }
  if (kt0 + 64 > sd.n_orig) {
    const int s_lo = max(kt0, sd.n_orig);
    const int off = s_lo - kt0;  // 0..63
    const uint64_t keep = off == 0 ? 0ull : ((1ull << off) - 1);
    vis = (vis & keep) | (bits_window(m.see_s, s_lo - sd.n_orig) << off);
  }
  return vis;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// AND of `ok` over the threads of named barrier `id` (`n` threads), which it also syncs.
__device__ __forceinline__ bool bar_and(int id, int n, bool ok) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
      "barrier.red.and.pred q, %2, %3, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(ok)), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

// Named barriers: 0 = __syncthreads, 1 = warps 0-3 (block info), 2 = the 8 softmax warps,
// then per kernel 3 + q (see the kernel).
__device__ __forceinline__ void softmax_bar_sync() {
  asm volatile("bar.sync 2, 256;" ::: "memory");
}
// The two softmax warps (q and q + 4) that share TMEM lane quarter q.
__device__ __forceinline__ void pair_bar_sync(int quarter) {
  asm volatile("bar.sync %0, 64;" ::"r"(3 + quarter) : "memory");
}


// ---------------------------------------------------------------- host side

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

bool make_map(CUtensorMap* m, const void* ptr, int heads, int d, int rows, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(heads) * d, static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(heads) * d * 2};
  const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// cudaFuncSetAttribute once per (kernel, device).
template <class F>
cudaError_t ensure_smem_attr(F* kernel, size_t bytes, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (done.load(std::memory_order_acquire) & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(bytes));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  if (e == cudaSuccess) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}
// Launch configuration of an attention kernel: an optional cluster of `cluster` CTAs along
// x, and programmatic dependent launch (pdl: the kernel may start while the RoPE key pass
// launched before it is still running; its producer waits for that pass before any key
// load). Not copyable: cfg points at attr.
struct AttnLaunch {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  AttnLaunch(unsigned grid, unsigned block, size_t smem, cudaStream_t stream, int cluster,
             bool pdl) {
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    int n = 0;
    if (cluster > 1) {
      attr[n].id = cudaLaunchAttributeClusterDimension;
      attr[n].val.clusterDim.x = cluster;
      attr[n].val.clusterDim.y = 1;
      attr[n].val.clusterDim.z = 1;
      ++n;
    }
    if (pdl) {
      attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[n].val.programmaticStreamSerializationAllowed = 1;
      ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
  }
  AttnLaunch(const AttnLaunch&) = delete;
  AttnLaunch& operator=(const AttnLaunch&) = delete;
};

int sm_count() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  int n = cache[dev].load(std::memory_order_relaxed);
  if (n <= 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    cache[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

}  // namespace
}  // namespace dard
