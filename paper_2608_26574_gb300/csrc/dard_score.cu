// dard_score.cu - confidence scoring and state transition of one DARD step (sm_103a).
//
// Implements Eq. 1 (max-probability and argmax), Eq. 5-6 (verification-outcome kernel and
// guidance weight), Eq. 7 (logit mixing) and Eq. 8 (three-state transition) in the order of
// Algorithm 1 of arXiv 2608.26574:
//
//   pass 1  rows in state C or U read their shadow logits once and are decided; C rows
//           record whether they were promoted (P) or demoted (D);
//   pass 2  rows in state M read both logit rows once, weight them by w from P and D of
//           their own block and are decided.
//
// Both passes split every vocabulary row over the `nsplit` CTAs of one thread-block
// cluster (256 threads each, 128-bit streaming loads, warp-shuffle merge of (max, sum of
// exp, argmax)). Each CTA writes its partial into the shared memory of the cluster's first
// CTA over DSMEM; after one cluster barrier that CTA merges the partials in split order
// (deterministic) and writes the row's outputs. Pass 2 is launched as a programmatic
// dependent of pass 1: its CTAs load their logits while pass 1 finishes and only then
// wait for pass 1's results. Pass 1 is itself a programmatic dependent of whatever kernel
// precedes the call and waits for it before touching memory.
//
// The number of CTAs per row follows the row count (split_cap). A compile-time variant
// (kExtra) adds the optional end-of-step outputs: p_cur, the next step's tokens, an
// in-place state update, entropy, margin and the next step's ordering key.
#include <atomic>
#include <cstdlib>
#include <cstring>
#include <type_traits>
#include <cfloat>
#include <climits>
#include <cmath>
#include <cstdio>

#include "dard_internal.h"
#include "dard_ptx.cuh"

namespace dard {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kWarps = kScoreThreads / 32;

struct Acc {
  float m;   // running maximum
  float s;   // sum of exp(x - m)
  int idx;   // lowest index attaining m
};

// Merge of two partial softmax summaries; equal maxima keep the lower index.
__device__ __forceinline__ Acc acc_merge(const Acc& a, const Acc& b) {
  const bool b_wins = (b.m > a.m) || (b.m == a.m && b.idx < a.idx);
  const Acc hi = b_wins ? b : a;
  const Acc lo = b_wins ? a : b;
  const float f = (lo.m == -INFINITY) ? 0.f : ex2_approx((lo.m - hi.m) * kLog2e);
  return {hi.m, fmaf(lo.s, f, hi.s), hi.idx};
}

__device__ __forceinline__ Acc warp_merge(Acc a) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Acc b;
    b.m = __shfl_xor_sync(0xffffffffu, a.m, off);
    b.s = __shfl_xor_sync(0xffffffffu, a.s, off);
    b.idx = __shfl_xor_sync(0xffffffffu, a.idx, off);
    a = acc_merge(a, b);
  }
  return a;
}

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// Element access for the two logit types; W elements per 16-byte vector.
struct Bf16 {
  static constexpr int W = 8;
  static constexpr int kBytes = 2;
  __device__ static float get(const uint4& v, int e) {
    const uint32_t w = (e >> 1) == 0 ? v.x : (e >> 1) == 1 ? v.y : (e >> 1) == 2 ? v.z : v.w;
    return __uint_as_float((e & 1) ? (w & 0xffff0000u) : (w << 16));
  }
  __device__ static float scalar(const char* p) {
    return __uint_as_float(static_cast<uint32_t>(*reinterpret_cast<const uint16_t*>(p)) << 16);
  }
};
struct F32 {
  static constexpr int W = 4;
  static constexpr int kBytes = 4;
  __device__ static float get(const uint4& v, int e) {
    const uint32_t w = e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
    return __uint_as_float(w);
  }
  __device__ static float scalar(const char* p) { return *reinterpret_cast<const float*>(p); }
};

constexpr uint32_t kNegInfBits = 0xff800000u;

// Loads vector v of this thread's round starting at element `base`; elements at or past c1
// read as -inf (neutral for max, argmax and the exp-sum).
template <class T>
__device__ __forceinline__ uint4 load_vec(const char* row, int e0, int c1) {
  if (e0 + T::W <= c1) return ld_stream(row + static_cast<size_t>(e0) * T::kBytes);
  uint4 r;
  uint32_t* w = &r.x;
  if (T::kBytes == 4) {
#pragma unroll
    for (int e = 0; e < 4; ++e)
      w[e] = (e0 + e < c1) ? __float_as_uint(T::scalar(row + static_cast<size_t>(e0 + e) * 4))
                           : kNegInfBits;
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int a = e0 + 2 * k, b = a + 1;
      const uint32_t lo = a < c1 ? *reinterpret_cast<const uint16_t*>(row + static_cast<size_t>(a) * 2)
                                 : (kNegInfBits >> 16);
      const uint32_t hi = b < c1 ? *reinterpret_cast<const uint16_t*>(row + static_cast<size_t>(b) * 2)
                                 : (kNegInfBits >> 16);
      w[k] = lo | (hi << 16);
    }
  }
  return r;
}

// Folds VPT*W values (given by `val(v, e)`, element index `base + (v*256 + tid)*W + e`) into
// the running accumulator: max/argmax first, then the exp-sum against the updated maximum.
// With kTail, elements at or past `limit` (padding of the last round) count as -inf.
template <class T, int VPT, bool kTail, class ValFn>
__device__ __forceinline__ void fold_round(Acc& acc, int base, int limit, ValFn val) {
  auto get = [&](int v, int e) {
    const float x = val(v, e);
    if (!kTail) return x;
    const int i = base + (v * kScoreThreads + static_cast<int>(threadIdx.x)) * T::W + e;
    return i < limit ? x : -INFINITY;
  };
  float m = -INFINITY;
  int idx = INT_MAX;
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
#pragma unroll
    for (int e = 0; e < T::W; ++e) {
      const float x = get(v, e);
      if (x > m) {
        m = x;
        idx = base + (v * kScoreThreads + static_cast<int>(threadIdx.x)) * T::W + e;
      }
    }
  }
  if (m > acc.m) {
    acc.s = (acc.m == -INFINITY) ? 0.f : acc.s * ex2_approx((acc.m - m) * kLog2e);
    acc.m = m;
    acc.idx = idx;
  }
  const float mL = (acc.m == -INFINITY) ? 0.f : acc.m * kLog2e;
  float s = 0.f;
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
#pragma unroll
    for (int e = 0; e < T::W; ++e) s += ex2_approx(fmaf(get(v, e), kLog2e, -mL));
  }
  acc.s += s;
}

template <class T, int VPT, class ValFn>
__device__ __forceinline__ void fold(Acc& acc, int base, int limit, ValFn val) {
  if (base + kScoreThreads * VPT * T::W <= limit) fold_round<T, VPT, false>(acc, base, limit, val);
  else fold_round<T, VPT, true>(acc, base, limit, val);
}

// Order-preserving map of non-NaN floats to unsigned integers (for redux.sync max).
__device__ __forceinline__ uint32_t order_key(float x) {
  const uint32_t b = __float_as_uint(x);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float from_key(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Warp-wide merge: maximum and argmax by redux.sync, then one rescale per lane and a
// shuffle tree for the sum (fixed order, so deterministic). m is never NaN (NaN values never
// win a comparison); a NaN sum propagates.
__device__ __forceinline__ Acc warp_merge_fast(const Acc& a) {
  const uint32_t key = order_key(a.m);
  const uint32_t kmax = __reduce_max_sync(0xffffffffu, key);
  const float mx = from_key(kmax);
  const uint32_t cand = key == kmax ? static_cast<uint32_t>(a.idx) : 0xffffffffu;
  const int idx = static_cast<int>(__reduce_min_sync(0xffffffffu, cand));
  const float f = (a.m == -INFINITY) ? 0.f : ex2_approx((a.m - mx) * kLog2e);
  float sum = a.s * f;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
  return {mx, sum, idx};
}

__device__ __forceinline__ Acc block_merge(Acc a, Acc* smem) {
  a = warp_merge_fast(a);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) smem[warp] = a;
  __syncthreads();
  if (warp == 0) {
    a = lane < kWarps ? smem[lane] : Acc{-INFINITY, 0.f, INT_MAX};
    a = warp_merge_fast(a);
  }
  return a;  // valid in warp 0
}

__device__ __forceinline__ int seq_of_row(const ScoreParams& p, int row) {
  int lo = 0, hi = p.num_seqs;  // blk_off[lo] <= row < blk_off[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.blk_off[mid] <= row) lo = mid; else hi = mid;
  }
  return lo;
}

__device__ __forceinline__ int load_state(const ScoreParams& p, int row, bool report) {
  int s = p.state_in[row];
  if (s > 2) {
    if (report && p.status) atomicOr(p.status, DARD_STATUS_BAD_STATE);
    s = kStateM;
  }
  return s;
}

// ---- the extended summary of the end-of-step variant: also hx = sum exp(x - m) x (the
// entropy sum is h = sum exp(x - m)(x - m) = hx - m s) and the second-largest value m2 (a
// repeated maximum counts as the second), for the entropy and margin of the ordering
// variants. Both rescale like s when the maximum grows.
struct AccX {
  float m;   // running maximum
  float s;   // sum of exp(x - m)
  int idx;   // lowest index attaining m
  float hx;  // sum of exp(x - m) * x
  float m2;  // second-largest value
};

__device__ __forceinline__ AccX accx_init() { return {-INFINITY, 0.f, INT_MAX, 0.f, -INFINITY}; }

// Warp-wide merge in the manner of warp_merge_fast; the second maximum is the largest of
// every lane's second value and of the first values of the lanes that do not hold the
// winning (maximum, lowest index) entry.
__device__ __forceinline__ AccX warp_merge_fast(const AccX& a) {
  const uint32_t key = order_key(a.m);
  const uint32_t kmax = __reduce_max_sync(0xffffffffu, key);
  const float mx = from_key(kmax);
  const uint32_t cand = key == kmax ? static_cast<uint32_t>(a.idx) : 0xffffffffu;
  const int idx = static_cast<int>(__reduce_min_sync(0xffffffffu, cand));
  const bool winner = key == kmax && a.idx == idx;
  const float c2 = winner ? a.m2 : fmaxf(a.m, a.m2);
  const float m2 = from_key(__reduce_max_sync(0xffffffffu, order_key(c2)));
  const float f = (a.m == -INFINITY) ? 0.f : ex2_approx((a.m - mx) * kLog2e);
  float sum = a.s * f, hx = a.hx * f;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    sum += __shfl_xor_sync(0xffffffffu, sum, off);
    hx += __shfl_xor_sync(0xffffffffu, hx, off);
  }
  return {mx, sum, idx, hx, m2};
}

template <class T, int VPT, bool kTail, class ValFn>
__device__ __forceinline__ void fold_round(AccX& acc, int base, int limit, ValFn val) {
  auto get = [&](int v, int e) {
    const float x = val(v, e);
    if (!kTail) return x;
    const int i = base + (v * kScoreThreads + static_cast<int>(threadIdx.x)) * T::W + e;
    return i < limit ? x : -INFINITY;
  };
  float m = -INFINITY, m2 = -INFINITY;
  int idx = INT_MAX;
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
#pragma unroll
    for (int e = 0; e < T::W; ++e) {
      const float x = get(v, e);
      m2 = fmaxf(m2, fminf(x, m));  // the old maximum, or x, becomes a second candidate
      if (x > m) {
        m = x;
        idx = base + (v * kScoreThreads + static_cast<int>(threadIdx.x)) * T::W + e;
      }
    }
  }
  acc.m2 = fmaxf(fmaxf(acc.m2, m2), fminf(acc.m, m));
  if (m > acc.m) {
    const float f = (acc.m == -INFINITY) ? 0.f : ex2_approx((acc.m - m) * kLog2e);
    acc.s *= f;
    acc.hx *= f;
    acc.m = m;
    acc.idx = idx;
  }
  if (acc.m == -INFINITY) return;
  const float mL = acc.m * kLog2e;
  float s = 0.f, hx = 0.f;
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
#pragma unroll
    for (int e = 0; e < T::W; ++e) {
      const float x = get(v, e);
      const float ex = ex2_approx(fmaf(x, kLog2e, -mL));
      s += ex;
      hx = fmaf(ex, fmaxf(x, -FLT_MAX), hx);  // -inf elements add 0, not NaN
    }
  }
  acc.s += s;
  acc.hx += hx;
}

template <class T, int VPT, class ValFn>
__device__ __forceinline__ void fold(AccX& acc, int base, int limit, ValFn val) {
  if (base + kScoreThreads * VPT * T::W <= limit) fold_round<T, VPT, false>(acc, base, limit, val);
  else fold_round<T, VPT, true>(acc, base, limit, val);
}

__device__ __forceinline__ AccX block_merge(AccX a, AccX* smem) {
  a = warp_merge_fast(a);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) smem[warp] = a;
  __syncthreads();
  if (warp == 0) {
    a = lane < kWarps ? smem[lane] : accx_init();
    a = warp_merge_fast(a);
  }
  return a;  // valid in warp 0
}

// Sends this CTA's partial (warp 0 holds it) to slot `split` of the leader CTA (cluster
// rank 0), then synchronises the cluster; afterwards the leader's slots are complete.
__device__ __forceinline__ void cluster_publish(const Acc& a, int split, float4* slots) {
  if (threadIdx.x == 0)
    st_cluster_v4(map_shared_rank(smem_u32(&slots[split]), 0), a.m, a.s, __int_as_float(a.idx),
                  0.f);
  cluster_sync();
}
// The extended summary uses the slot pair (split, kScoreMaxSplit + split).
__device__ __forceinline__ void cluster_publish(const AccX& a, int split, float4* slots) {
  if (threadIdx.x == 0) {
    st_cluster_v4(map_shared_rank(smem_u32(&slots[split]), 0), a.m, a.s, __int_as_float(a.idx),
                  a.hx);
    st_cluster_v4(map_shared_rank(smem_u32(&slots[kScoreMaxSplit + split]), 0), a.m2, 0.f, 0.f,
                  0.f);
  }
  cluster_sync();
}

// Merges the leader's slots in split order (warp 0); returns the row summary in lane 0.
__device__ __forceinline__ void merge_slots(const float4* slots, int nsplit, Acc& out) {
  Acc a{-INFINITY, 0.f, INT_MAX};
  const int lane = threadIdx.x & 31;
  if (lane < nsplit) {
    const float4 v = slots[lane];
    a = Acc{v.x, v.y, __float_as_int(v.z)};
  }
  out = warp_merge(a);
}
__device__ __forceinline__ void merge_slots(const float4* slots, int nsplit, AccX& out) {
  AccX a = accx_init();
  const int lane = threadIdx.x & 31;
  if (lane < nsplit) {
    const float4 v = slots[lane], v2 = slots[kScoreMaxSplit + lane];
    a = AccX{v.x, v.y, __float_as_int(v.z), v.w, v2.x};
  }
  out = warp_merge_fast(a);
}

__device__ __forceinline__ Acc acc_init(Acc*) { return {-INFINITY, 0.f, INT_MAX}; }
__device__ __forceinline__ AccX acc_init(AccX*) { return accx_init(); }

// The current token's logits (for p_cur), loaded by the leader's thread 0 when the CTA
// starts so that their latency hides behind the row's stream; -inf marks "no token".
template <class T>
__device__ __forceinline__ void prefetch_current(const ScoreParams& p, int row, const char* xp,
                                                 const char* sp, float& lx, float& ls) {
  lx = ls = -INFINITY;
  if (p.p_cur == nullptr || threadIdx.x != 0 || blockIdx.x != 0) return;
  const int ct = p.cur_token[row];
  if (ct < 0 || ct >= p.vocab) return;
  const size_t off = static_cast<size_t>(ct) * T::kBytes;
  ls = T::scalar(sp + off);
  if (xp) lx = T::scalar(xp + off);
}

// Eq. 1 and Eq. 8 on a merged row; writes conf / token / state, the optional p_cur (of the
// current token's scored logit lc) and next-step token (x^, or the mask token for a row
// that ends in M: the last line of Algorithm 1's step); returns the new state.
template <bool kExtra, class A>
__device__ __forceinline__ int finalize_row(const ScoreParams& p, int row, const A& a,
                                            float w, float lc, bool write_state = true) {
  const float z = a.s;
  const bool valid = isfinite(z) && z > 0.f;
  const float c = valid ? 1.0f / z : 0.f;
  const int ns = !valid ? kStateM : (c <= p.tau_c ? kStateM : (c <= p.tau_u ? kStateC : kStateU));
  p.conf[row] = c;
  p.token[row] = valid ? a.idx : -1;
  if (write_state) p.state_out[row] = static_cast<uint8_t>(ns);
  if (p.w_out) p.w_out[row] = w;
  if (kExtra && p.p_cur) {
    const float mL = a.m * kLog2e;
    p.p_cur[row] = (valid && lc != -INFINITY) ? ex2_approx(fmaf(lc, kLog2e, -mL)) / z : 0.f;
  }
  if (kExtra && p.tokens) p.tokens[row] = ns == kStateM ? p.mask_token : a.idx;
  if constexpr (kExtra) {
    // entropy (nats) and margin of the scored distribution, the next step's ordering key
    const float hnat = valid ? logf(z) + a.m - a.hx / z : 0.f;  // ln Z - (hx - m Z) / Z
    const float mg = valid ? (1.0f - ex2_approx((a.m2 - a.m) * kLog2e)) / z : 0.f;
    if (p.entropy) p.entropy[row] = hnat;
    if (p.margin) p.margin[row] = mg;
    if (p.order_key) {
      const int i = row - p.blk_off[seq_of_row(p, row)];
      p.order_key[row] = p.order_mode == DARD_ORDER_BIDIR ? 0.f
                       : p.order_mode == DARD_ORDER_L2R ? -static_cast<float>(i)
                       : p.order_mode == DARD_ORDER_ENTROPY ? -hnat
                       : p.order_mode == DARD_ORDER_MARGIN ? mg : c;
    }
  }
  if (!valid && p.status) atomicOr(p.status, DARD_STATUS_INVALID_ROW);
  return ns;
}

// M/C/U counts of every sequence: zeroed by one thread of pass 1, then every row adds its
// final state in pass 2 (after the grid dependency, so the zeroing is visible).
__device__ __forceinline__ void zero_counts(const ScoreParams& p) {
  if (p.counts != nullptr && blockIdx.x == 0 && blockIdx.y == 0)
    for (int k = threadIdx.x; k < 3 * p.num_seqs; k += blockDim.x) p.counts[k] = 0;
}
__device__ __forceinline__ void add_count(const ScoreParams& p, int seq, int state) {
  if (p.counts != nullptr) atomicAdd(&p.counts[seq * 3 + state], 1);
}

// kExtra: the call asks for p_cur, next-step tokens or an in-place state update.
template <class T, int VPT, bool kExtra>
__global__ void __launch_bounds__(kScoreThreads) score_pass1(const __grid_constant__ ScoreParams p) {
  // Launched with programmatic dependent launch after whatever kernel precedes the call
  // (the LM head in a model, the attention kernel in the benchmark): this CTA may already be
  // resident, but it touches no memory before that kernel has completed. Only then may
  // pass 2 start: it loads its logits (and the states) before it waits for pass 1, so
  // the kernel that wrote them must have completed by the time pass 2 is launched, even
  // when that kernel lets its own dependents start early.
  grid_dep_wait();
  grid_dep_launch();
  using A = std::conditional_t<kExtra, AccX, Acc>;
  __shared__ A s_acc[kWarps];
  __shared__ float4 s_slots[2 * kScoreMaxSplit];
  zero_counts(p);
  const int row = blockIdx.y, split = blockIdx.x;  // split = rank in the row's cluster
  const int st = load_state(p, row, split == 0);
  if (st == kStateM) {  // uniform over the cluster: no CTA of it reaches the barrier
    if (split == 0) p.pd_flag[row] = 3;  // pass 2's row (even if state_out overwrites it)
    return;
  }
  const char* rowp = static_cast<const char*>(p.ls) + static_cast<size_t>(row) * p.row_stride * T::kBytes;
  const int c0 = split * p.chunk;
  const int c1 = min(p.vocab, c0 + p.chunk);
  float cur_lx = 0.f, cur_ls = 0.f;  // the current token's logit (p_cur), loaded early
  if (kExtra) prefetch_current<T>(p, row, nullptr, rowp, cur_lx, cur_ls);
  A acc = acc_init(static_cast<A*>(nullptr));
  for (int base = c0; base < c1; base += kScoreThreads * VPT * T::W) {
    uint4 r[VPT];
#pragma unroll
    for (int v = 0; v < VPT; ++v)
      r[v] = load_vec<T>(rowp, base + (v * kScoreThreads + threadIdx.x) * T::W, c1);
    fold<T, VPT>(acc, base, c1, [&](int v, int e) { return T::get(r[v], e); });
  }
  acc = block_merge(acc, s_acc);
  cluster_publish(acc, split, s_slots);
  if (split != 0 || threadIdx.x >= 32) return;
  A a;
  merge_slots(s_slots, p.nsplit, a);
  if (threadIdx.x == 0) {
    const int ns = finalize_row<kExtra>(p, row, a, __int_as_float(0x7fc00000), cur_ls);
    p.pd_flag[row] = (st == kStateC) ? (ns == kStateU ? 1 : (ns == kStateM ? 2 : 0)) : 0;
  }
}

template <class T, int VPT, bool kExtra>
__global__ void __launch_bounds__(kScoreThreads) score_pass2(const __grid_constant__ ScoreParams p) {
  using A = std::conditional_t<kExtra, AccX, Acc>;
  __shared__ A s_acc[kWarps];
  __shared__ float4 s_slots[2 * kScoreMaxSplit];
  __shared__ float s_w;
  __shared__ bool s_m_row;
  const int row = blockIdx.y, split = blockIdx.x;
  const int st = load_state(p, row, false);
  const int seq = seq_of_row(p, row);
  if (st != kStateM) {
    // The first row's first CTA waits for pass 1 even when nothing is counted, so that this
    // grid cannot end before pass 1 has (also when no row is M): the call's last kernel
    // ends after all of the call's work.
    if (split == 0 && threadIdx.x == 0 && (p.counts != nullptr || row == 0)) {
      grid_dep_wait();
      if (p.counts != nullptr) add_count(p, seq, __ldcg(p.state_out + row));
    }
    return;
  }
  const size_t roff = static_cast<size_t>(row) * p.row_stride * T::kBytes;
  const char* xp = static_cast<const char*>(p.lx) + roff;
  const char* sp = static_cast<const char*>(p.ls) + roff;
  const int c0 = split * p.chunk;
  const int c1 = min(p.vocab, c0 + p.chunk);
  float cur_lx = 0.f, cur_ls = 0.f;  // the current token's logits (p_cur), loaded early
  if (kExtra) prefetch_current<T>(p, row, xp, sp, cur_lx, cur_ls);

  // The first round's loads do not depend on pass 1: issue them before waiting for it.
  uint4 rx[VPT], rs[VPT];
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    const int e0 = c0 + (v * kScoreThreads + threadIdx.x) * T::W;
    rx[v] = load_vec<T>(xp, e0, c1);
    rs[v] = load_vec<T>(sp, e0, c1);
  }
  grid_dep_wait();

  // Eq. 5-6: w from the verification outcomes of this block, computed by warp 0: each lane
  // sums lambda^|i-j| = 2^(|i-j| log2 lambda) over its positions, then a shuffle tree.
  // With state_out aliasing state_in, a C or U row that pass 1 moved to M reads as M above;
  // its own outcome byte (3 = an M row), loaded beside the others, tells them apart (only
  // then: without aliasing the state read above is this step's).
  const int b0 = p.blk_off[seq], blen = p.blk_off[seq + 1] - b0;
  const int i = row - b0;
  if (threadIdx.x < 32) {
    const int own = (kExtra && threadIdx.x == 0 && p.state_in_place) ? __ldcg(p.pd_flag + row) : 3;
    float pp = 0.f, dd = 0.f;
    for (int j = threadIdx.x; j < blen; j += 32) {
      const int f = __ldcg(p.pd_flag + b0 + j);
      const float kij = ex2_approx(static_cast<float>(abs(i - j)) * p.log2_lambda);
      pp += f == 1 ? kij : 0.f;
      dd += f == 2 ? kij : 0.f;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      pp += __shfl_xor_sync(0xffffffffu, pp, off);
      dd += __shfl_xor_sync(0xffffffffu, dd, off);
    }
    if (threadIdx.x == 0) {
      s_w = __fdiv_rn(pp + p.p0, pp + dd + p.p0);
      if (kExtra) s_m_row = own == 3;
    }
  }
  __syncthreads();
  if (kExtra && !s_m_row) {  // uniform over the cluster
    if (split == 0 && p.counts != nullptr && threadIdx.x == 0)
      add_count(p, seq, __ldcg(p.state_out + row));
    return;
  }
  const float w = s_w;

  // Eq. 7 in fp32, one rounding per operation: mix = ls + w * (lx - ls).
  auto mix = [&](const uint4& vx, const uint4& vs, int e) {
    const float lx = T::get(vx, e), ls = T::get(vs, e);
    return __fadd_rn(ls, __fmul_rn(w, __fsub_rn(lx, ls)));
  };
  A acc = acc_init(static_cast<A*>(nullptr));
  fold<T, VPT>(acc, c0, c1, [&](int v, int e) { return mix(rx[v], rs[v], e); });
  for (int base = c0 + kScoreThreads * VPT * T::W; base < c1; base += kScoreThreads * VPT * T::W) {
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int e0 = base + (v * kScoreThreads + threadIdx.x) * T::W;
      rx[v] = load_vec<T>(xp, e0, c1);
      rs[v] = load_vec<T>(sp, e0, c1);
    }
    fold<T, VPT>(acc, base, c1, [&](int v, int e) { return mix(rx[v], rs[v], e); });
  }
  acc = block_merge(acc, s_acc);
  cluster_publish(acc, split, s_slots);
  if (split != 0 || threadIdx.x >= 32) return;
  A a;
  merge_slots(s_slots, p.nsplit, a);
  if (threadIdx.x == 0) {
    const float lc = cur_ls == -INFINITY ? -INFINITY
                                         : __fadd_rn(cur_ls, __fmul_rn(w, __fsub_rn(cur_lx, cur_ls)));
    add_count(p, seq, finalize_row<kExtra>(p, row, a, w, lc));
  }
}

// ------------------------------------------------------------------ one-launch scoring
// Both passes in one grid. C and U rows stream their shadow logits and decide (Eq. 1, 8);
// a C row's cluster leader then writes its outcome byte and releases the block's ready
// counter. M rows issue the loads of their first round of both logit rows, wait until
// every C row of their block has published (a bounded spin on the counter: the launcher
// uses this kernel only when the whole grid fits on the device at once, so every C row
// the wait depends on is running), compute w (Eq. 5-6) and mix (Eq. 7).
// Counters start at zero and every call leaves them at zero: the last M-row CTA of a
// block to pass its wait clears ready and departed; with counts or an in-place state
// update, the last row of a block to finish (fin) writes the block's counts and states
// and clears fin.

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_gpu(uint32_t* p, uint32_t v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

template <class T, int VPT, bool kExtra>
__global__ void __launch_bounds__(kScoreThreads) score_fused(const __grid_constant__ ScoreParams p) {
  // Launched as a programmatic dependent of whatever kernel precedes the call: nothing is
  // read before that kernel (the logits' producer, or the previous call that leaves the
  // counters at zero) has completed.
  grid_dep_wait();
  using A = std::conditional_t<kExtra, AccX, Acc>;
  __shared__ A s_acc[kWarps];
  __shared__ float4 s_slots[2 * kScoreMaxSplit];
  __shared__ float s_w;
  __shared__ int s_nm;
  if (p.counts != nullptr && blockIdx.x == 0 && blockIdx.y == 0) {
    // sequences with an empty block have no row to write their counts
    for (int k = threadIdx.x; k < p.num_seqs; k += blockDim.x)
      if (p.blk_off[k + 1] == p.blk_off[k]) {
        p.counts[3 * k + 0] = 0;
        p.counts[3 * k + 1] = 0;
        p.counts[3 * k + 2] = 0;
      }
  }
  const int row = blockIdx.y, split = blockIdx.x;
  const int seq = seq_of_row(p, row);
  const int b0 = p.blk_off[seq], blen = p.blk_off[seq + 1] - b0;
  const int st = load_state(p, row, split == 0);
  const size_t roff = static_cast<size_t>(row) * p.row_stride * T::kBytes;
  const char* xp = static_cast<const char*>(p.lx) + roff;
  const char* sp = static_cast<const char*>(p.ls) + roff;
  const int c0 = split * p.chunk;
  const int c1 = min(p.vocab, c0 + p.chunk);
  float cur_lx = 0.f, cur_ls = 0.f;  // the current token's logits (p_cur), loaded early
  if (kExtra) prefetch_current<T>(p, row, st == kStateM ? xp : nullptr, sp, cur_lx, cur_ls);
  A acc = acc_init(static_cast<A*>(nullptr));
  float w = __int_as_float(0x7fc00000);
  constexpr int kRound = kScoreThreads * VPT * T::W;
  if (st != kStateM) {
    // The block's M count (a C row releases the counter only if some M row waits on it).
    if (threadIdx.x < 32) {
      int nm = 0;
      for (int j = threadIdx.x; j < blen; j += 32) {
        const int sj = p.state_in[b0 + j];
        nm += (sj == kStateM || sj > 2) ? 1 : 0;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) nm += __shfl_xor_sync(0xffffffffu, nm, off);
      if (threadIdx.x == 0) s_nm = nm;
    }
    for (int base = c0; base < c1; base += kRound) {
      uint4 r[VPT];
#pragma unroll
      for (int v = 0; v < VPT; ++v)
        r[v] = load_vec<T>(sp, base + (v * kScoreThreads + threadIdx.x) * T::W, c1);
      fold<T, VPT>(acc, base, c1, [&](int v, int e) { return T::get(r[v], e); });
    }
  } else {
    // First round of both rows: in flight while the block's C rows are decided.
    uint4 rx[VPT], rs[VPT];
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int e0 = c0 + (v * kScoreThreads + threadIdx.x) * T::W;
      rx[v] = load_vec<T>(xp, e0, c1);
      rs[v] = load_vec<T>(sp, e0, c1);
    }
    if (threadIdx.x < 32) {
      const int lane = threadIdx.x;
      int nc = 0, nm = 0;
      for (int j = lane; j < blen; j += 32) {
        const int sj = p.state_in[b0 + j];
        nc += sj == kStateC ? 1 : 0;
        nm += (sj == kStateM || sj > 2) ? 1 : 0;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        nc += __shfl_xor_sync(0xffffffffu, nc, off);
        nm += __shfl_xor_sync(0xffffffffu, nm, off);
      }
      bool ok = true;
      if (nc > 0) {
        if (lane == 0) {
          const uint32_t need = static_cast<uint32_t>(nc);
          if (ld_acquire_gpu(p.ready + seq) < need) {
            const long long t0 = clock64();
            while (ld_acquire_gpu(p.ready + seq) < need) {
              if (clock64() - t0 > kWaitCycles) { ok = false; break; }
              __nanosleep(64);
            }
          }
          if (!ok && p.status) atomicOr(p.status, DARD_STATUS_TIMEOUT);
        }
        __syncwarp();
        (void)ld_acquire_gpu(p.ready + seq);  // this lane's own acquire before the reads below
      }
      // Eq. 5-6 from the outcome bytes of this step's C rows: lambda^|i-j| as
      // 2^(|i-j| log2 lambda), fp32 sums over the lanes, then a shuffle tree.
      const int i = row - b0;
      float pp = 0.f, dd = 0.f;
      for (int j = lane; j < blen && nc > 0; j += 32) {
        if (p.state_in[b0 + j] != kStateC) continue;
        const int f = *reinterpret_cast<volatile const uint8_t*>(p.pd_flag + b0 + j);
        const float kij = ex2_approx(static_cast<float>(abs(i - j)) * p.log2_lambda);
        pp += f == 1 ? kij : 0.f;
        dd += f == 2 ? kij : 0.f;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        pp += __shfl_xor_sync(0xffffffffu, pp, off);
        dd += __shfl_xor_sync(0xffffffffu, dd, off);
      }
      if (lane == 0) {
        s_w = __fdiv_rn(pp + p.p0, pp + dd + p.p0);
        // the last M-row CTA of the block past its wait clears the block's counters
        if (nc > 0) {
          const uint32_t leaving = atomicAdd(p.departed + seq, 1u) + 1u;
          if (leaving == static_cast<uint32_t>(nm * p.nsplit)) {
            p.ready[seq] = 0;
            p.departed[seq] = 0;
          }
        }
      }
    }
    __syncthreads();
    w = s_w;
    // Eq. 7 in fp32, one rounding per operation: mix = ls + w * (lx - ls).
    auto mix = [&](const uint4& vx, const uint4& vs, int e) {
      const float lx = T::get(vx, e), ls = T::get(vs, e);
      return __fadd_rn(ls, __fmul_rn(w, __fsub_rn(lx, ls)));
    };
    fold<T, VPT>(acc, c0, c1, [&](int v, int e) { return mix(rx[v], rs[v], e); });
    for (int base = c0 + kRound; base < c1; base += kRound) {
#pragma unroll
      for (int v = 0; v < VPT; ++v) {
        const int e0 = base + (v * kScoreThreads + threadIdx.x) * T::W;
        rx[v] = load_vec<T>(xp, e0, c1);
        rs[v] = load_vec<T>(sp, e0, c1);
      }
      fold<T, VPT>(acc, base, c1, [&](int v, int e) { return mix(rx[v], rs[v], e); });
    }
  }
  acc = block_merge(acc, s_acc);
  cluster_publish(acc, split, s_slots);
  if (split != 0 || threadIdx.x >= 32) return;
  A a;
  merge_slots(s_slots, p.nsplit, a);
  if (threadIdx.x != 0) return;
  float lc = cur_ls;
  if (st == kStateM && cur_ls != -INFINITY)
    lc = __fadd_rn(cur_ls, __fmul_rn(w, __fsub_rn(cur_lx, cur_ls)));
  // in place, the block's states are written by its last row (the others may still read them)
  const int ns = finalize_row<kExtra>(p, row, a, w, lc, !p.state_in_place);
  if (st == kStateC && s_nm > 0) {
    // the outcome byte, then the release of the block's counter (Algorithm 1: P and D)
    p.pd_flag[row] = ns == kStateU ? 1 : (ns == kStateM ? 2 : 0);
    red_release_gpu(p.ready + seq, 1u);
  }
  if (p.counts != nullptr || p.state_in_place) {
    p.new_state[row] = static_cast<uint8_t>(ns);
    __threadfence();
    if (atomicAdd(p.fin + seq, 1u) + 1u == static_cast<uint32_t>(blen)) {
      // the block's last row: every row of it has read its states and written new_state
      __threadfence();
      int cnt[3] = {0, 0, 0};
      for (int j = 0; j < blen; ++j) {
        const int nsj = *reinterpret_cast<volatile const uint8_t*>(p.new_state + b0 + j);
        cnt[nsj] += 1;
        if (p.state_in_place) p.state_out[b0 + j] = static_cast<uint8_t>(nsj);
      }
      if (p.counts != nullptr) {
        p.counts[3 * seq + 0] = cnt[0];
        p.counts[3 * seq + 1] = cnt[1];
        p.counts[3 * seq + 2] = cnt[2];
      }
      p.fin[seq] = 0;
    }
  }
}

// Zeroes the counts when there are no rows at all (no pass runs).
__global__ void zero_all_counts(const __grid_constant__ ScoreParams p) {
  for (int k = threadIdx.x; k < 3 * p.num_seqs; k += blockDim.x) p.counts[k] = 0;
}

template <class F>
cudaError_t allow_wide_clusters(F* kernel, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (done.load(std::memory_order_acquire) & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// Clusters of nsplit CTAs of this kernel that fit on the current device at once (cached
// per device and cluster size).
template <class K>
int max_active_clusters(K* kernel, int nsplit) {
  static std::atomic<int> cache[64][kScoreMaxSplit + 1];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64 || nsplit < 1 ||
      nsplit > kScoreMaxSplit)
    return 0;
  int n = cache[dev][nsplit].load(std::memory_order_relaxed);
  if (n > 0) return n;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nsplit, 1);
  cfg.blockDim = dim3(kScoreThreads);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = nsplit;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return 0;
  }
  cache[dev][nsplit].store(n, std::memory_order_relaxed);
  return n;
}

template <class T, int VPT, bool kExtra>
cudaError_t launch_fused(const ScoreParams& p, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.nsplit, p.rows);
  cfg.blockDim = dim3(kScoreThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.nsplit;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, score_fused<T, VPT, kExtra>, p);
}

template <class T, int VPT, bool kExtra>
cudaError_t launch_pair(const ScoreParams& p, cudaStream_t stream) {
  static std::atomic<uint64_t> done1{0}, done2{0};
  cudaError_t e = allow_wide_clusters(score_pass1<T, VPT, kExtra>, done1);
  if (e == cudaSuccess) e = allow_wide_clusters(score_pass2<T, VPT, kExtra>, done2);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.nsplit, p.rows);
  cfg.blockDim = dim3(kScoreThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.nsplit;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, score_pass1<T, VPT, kExtra>, p);
  if (e != cudaSuccess) return e;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, score_pass2<T, VPT, kExtra>, p);
}

}  // namespace

// Workspace: per-sequence counters (ready, departed, fin: zero between calls), then one
// outcome byte and one new-state byte per block row, each part 256-byte aligned.
namespace {
size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }
}  // namespace

size_t score_workspace_bytes(int32_t rows, int32_t num_seqs) {
  return align256(3 * sizeof(uint32_t) * static_cast<size_t>(num_seqs)) +
         2 * align256(static_cast<size_t>(rows));
}

size_t score_counter_bytes(int32_t num_seqs) {
  return align256(3 * sizeof(uint32_t) * static_cast<size_t>(num_seqs));
}

namespace {

// Number of SMs of the current device (looked up once per device).
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

// CTAs per row: few rows spread over up to kScoreMaxSplit CTAs so that the call still has
// about kScoreCtasPerSm CTAs per SM in flight; many rows get one or a few CTAs each, every
// CTA then streaming more rounds of its row (fewer merges, deeper per-CTA pipelines).
int split_cap(int rows) {
  const long long want = (static_cast<long long>(kScoreCtasPerSm) * sm_count() + rows - 1) /
                         std::max(rows, 1);
  return static_cast<int>(std::max(1ll, std::min<long long>(kScoreMaxSplit, want)));
}

}  // namespace

namespace {

// Splits every row over at most `cap` CTAs: each takes `rounds` rounds of 256 threads x 4
// vectors.
void set_split(ScoreParams& p, int per_round, int cap) {
  const int rounds_total = (p.vocab + per_round - 1) / per_round;
  const int rounds = (rounds_total + cap - 1) / cap;
  p.chunk = per_round * rounds;
  p.nsplit = (p.vocab + p.chunk - 1) / p.chunk;
}

// The two PDL-chained passes; with DARD_SCORE_PATH=fused, the one-launch kernel instead when
// every row's cluster fits on the device at once (its M rows wait for C rows of the same
// launch), with as many CTAs per row as allows that. Measured on GB300 (CUDA-graph timing,
// one call per input set): the passes take 8.3 us on the 8B block, 13.5 us on the GQA block,
// 25 us on the multimodal batch; the one launch 11.9, 18.4 and 34 us (10.4, 16.2 with no
// counts requested). The pass boundary is a completed grid, which the hardware signals
// sooner than the counters in L2 that the one launch polls.
template <class T, bool kExtra>
cudaError_t launch_rows(ScoreParams& p, cudaStream_t stream, int per_round) {
  static std::atomic<uint64_t> done{0};
  const char* force = std::getenv("DARD_SCORE_PATH");
  const bool fused = force != nullptr && std::strcmp(force, "fused") == 0;
  if (fused && allow_wide_clusters(score_fused<T, 4, kExtra>, done) == cudaSuccess) {
    const ScoreParams keep = p;
    for (int cap = p.nsplit; cap >= 1; --cap) {
      set_split(p, per_round, cap);
      if (max_active_clusters(score_fused<T, 4, kExtra>, p.nsplit) >= p.rows)
        return launch_fused<T, 4, kExtra>(p, stream);
      cap = p.nsplit;  // the next smaller split
    }
    p = keep;
  }
  return launch_pair<T, 4, kExtra>(p, stream);
}

}  // namespace

dard_status launch_score(const dard_score_args& a, ScoreParams& p, cudaStream_t stream,
                         char* err, size_t err_len) {
  const bool bf16 = a.dtype == DARD_BF16;
  const int W = bf16 ? 8 : 4;
  const int per_round = kScoreThreads * 4 * W;
  set_split(p, per_round, split_cap(p.rows));

  char* ws = static_cast<char*>(a.workspace);
  const size_t cbytes = score_counter_bytes(p.num_seqs);
  p.ready = reinterpret_cast<uint32_t*>(ws);
  p.departed = p.ready + p.num_seqs;
  p.fin = p.departed + p.num_seqs;
  p.pd_flag = reinterpret_cast<uint8_t*>(ws + cbytes);
  p.new_state = p.pd_flag + align256(static_cast<size_t>(p.rows));
  p.log2_lambda = static_cast<float>(std::log2(static_cast<double>(p.lambda)));

  // Test hook (failure-path tests; unset in normal operation): a launch that reports
  // failure without launching.
  if (std::getenv("DARD_TEST_FAIL_LAUNCH") != nullptr) {
    snprintf(err, err_len, "scoring launch failed: %s (DARD_TEST_FAIL_LAUNCH)",
             cudaGetErrorString(cudaErrorLaunchFailure));
    return DARD_ERR_CUDA;
  }
  cudaError_t e = cudaSuccess;
  if (p.counts != nullptr && p.rows == 0) {
    zero_all_counts<<<1, 256, 0, stream>>>(p);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess && p.rows > 0) {
    const bool extra = p.p_cur != nullptr || p.tokens != nullptr || p.state_in_place ||
                       p.entropy != nullptr || p.margin != nullptr || p.order_key != nullptr;
    if (extra) e = bf16 ? launch_rows<Bf16, true>(p, stream, per_round)
                        : launch_rows<F32, true>(p, stream, per_round);
    else e = bf16 ? launch_rows<Bf16, false>(p, stream, per_round)
                  : launch_rows<F32, false>(p, stream, per_round);
  }
  if (e != cudaSuccess) {
    snprintf(err, err_len, "scoring launch failed: %s", cudaGetErrorString(e));
    return DARD_ERR_CUDA;
  }
  return DARD_OK;
}

}  // namespace dard
