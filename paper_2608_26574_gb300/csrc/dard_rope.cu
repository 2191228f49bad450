// dard_rope.cu - the RoPE pass over the key rows of an attention call (rope_theta > 0).
//
// Every key row is read by every query tile of its sequence and every query head of its
// group, so the keys are rotated once here, into k_rope, rather than in each CTA that loads
// them; the attention kernel launched next on the stream waits for this grid
// (griddepcontrol) before its first key load, and rotates its own query tiles as it loads
// them. Positions and arithmetic: dard_rope.cuh.
//
// One thread per (row, group of four frequencies, four heads): the four cos/sin pairs are
// formed once and applied to the thread's elements of each of its heads. Interleaved
// pairing: a group is eight consecutive elements; half pairing: four elements of the first
// half and the four D/2 later. Consecutive threads take consecutive groups of one row and
// head, so a warp reads and writes whole 16-byte runs.
#include <cuda_bf16.h>

#include "dard_ptx.cuh"
#include "dard_rope.cuh"

namespace dard {
namespace {

constexpr int kRopeThreads = 256;
constexpr int kRopeHeads = 4;  // heads per thread

// Sequence of global row `row` (rows are stored sequence after sequence).
__device__ __forceinline__ int seq_of_row(const AttnParams& p, int row) {
  int lo = 0, hi = p.num_seqs - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.seq[mid].row_base <= row) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

__device__ __forceinline__ void rot(float& a, float& b, float c, float s) {
  const float x = a, y = b;
  a = fmaf(x, c, -y * s);
  b = fmaf(x, s, y * c);
}

template <typename T, int D>
__global__ void __launch_bounds__(kRopeThreads) rope_keys(const __grid_constant__ AttnParams p) {
  grid_dep_launch();  // the attention kernel may be scheduled; it waits for this grid's end
  constexpr int kGroups = D / 8;  // groups of four frequencies per row
  const int hblocks = (p.hkv + kRopeHeads - 1) / kRopeHeads;
  const long long idx = static_cast<long long>(blockIdx.x) * kRopeThreads + threadIdx.x;
  const long long total = static_cast<long long>(p.total_rows) * hblocks * kGroups;
  if (idx >= total) return;
  const int grp = static_cast<int>(idx % kGroups);
  const long long rest = idx / kGroups;
  const int hb = static_cast<int>(rest % hblocks);
  const int row = static_cast<int>(rest / hblocks);
  const SeqDesc& sd = p.seq[seq_of_row(p, row)];
  const int pos = rope_position(p, sd, row - sd.row_base);
  const bool half = p.rope_style == DARD_ROPE_HALF;
  // element offsets of the group within a head: [e0, e0 + 4) and [e1, e1 + 4)
  const int e0 = half ? 4 * grp : 8 * grp;
  const int e1 = half ? D / 2 + 4 * grp : 8 * grp + 4;
  const T* src = static_cast<const T*>(p.k_src);
  T* dst = static_cast<T*>(const_cast<void*>(p.k));
  const int h0 = hb * kRopeHeads;
  // every head's loads first (they are independent), then the rotations and the stores
  float x[kRopeHeads][8];
#pragma unroll
  for (int hh = 0; hh < kRopeHeads; ++hh) {
    if (h0 + hh >= p.hkv) break;
    const size_t base = (static_cast<size_t>(row) * p.hkv + h0 + hh) * D;
    if constexpr (sizeof(T) == 2) {
      const uint2 u0 = *reinterpret_cast<const uint2*>(src + base + e0);
      const uint2 u1 = *reinterpret_cast<const uint2*>(src + base + e1);
      x[hh][0] = bf_lo(u0.x); x[hh][1] = bf_hi(u0.x); x[hh][2] = bf_lo(u0.y); x[hh][3] = bf_hi(u0.y);
      x[hh][4] = bf_lo(u1.x); x[hh][5] = bf_hi(u1.x); x[hh][6] = bf_lo(u1.y); x[hh][7] = bf_hi(u1.y);
    } else {
      const float4 u0 = *reinterpret_cast<const float4*>(src + base + e0);
      const float4 u1 = *reinterpret_cast<const float4*>(src + base + e1);
      x[hh][0] = u0.x; x[hh][1] = u0.y; x[hh][2] = u0.z; x[hh][3] = u0.w;
      x[hh][4] = u1.x; x[hh][5] = u1.y; x[hh][6] = u1.z; x[hh][7] = u1.w;
    }
  }
  // the angles while the loads are in flight
  float c[4], s[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int i = 4 * grp + e;  // frequency index
    rope_cos_sin(pos, p.rope_f[2 * i], p.rope_f[2 * i + 1], c[e], s[e]);
  }
#pragma unroll
  for (int hh = 0; hh < kRopeHeads; ++hh) {
    if (h0 + hh >= p.hkv) break;
    float* y = x[hh];
    if (half) {
#pragma unroll
      for (int e = 0; e < 4; ++e) rot(y[e], y[4 + e], c[e], s[e]);
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) rot(y[2 * e], y[2 * e + 1], c[e], s[e]);
    }
    const size_t base = (static_cast<size_t>(row) * p.hkv + h0 + hh) * D;
    if constexpr (sizeof(T) == 2) {
      *reinterpret_cast<uint2*>(dst + base + e0) = make_uint2(bf_pack(y[0], y[1]), bf_pack(y[2], y[3]));
      *reinterpret_cast<uint2*>(dst + base + e1) = make_uint2(bf_pack(y[4], y[5]), bf_pack(y[6], y[7]));
    } else {
      *reinterpret_cast<float4*>(dst + base + e0) = make_float4(y[0], y[1], y[2], y[3]);
      *reinterpret_cast<float4*>(dst + base + e1) = make_float4(y[4], y[5], y[6], y[7]);
    }
  }
}

template <typename T>
cudaError_t launch_typed(const AttnParams& p, cudaStream_t stream) {
  const long long hblocks = (p.hkv + kRopeHeads - 1) / kRopeHeads;
  const long long threads = static_cast<long long>(p.total_rows) * hblocks * (p.head_dim / 8);
  const long long blocks = (threads + kRopeThreads - 1) / kRopeThreads;
  if (blocks < 1) return cudaSuccess;
  if (blocks > 0x7fffffffll) return cudaErrorInvalidValue;
  if (p.head_dim == 64)
    rope_keys<T, 64><<<static_cast<unsigned>(blocks), kRopeThreads, 0, stream>>>(p);
  else
    rope_keys<T, 128><<<static_cast<unsigned>(blocks), kRopeThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rope_keys(const AttnParams& p, int dtype, cudaStream_t stream) {
  return dtype == DARD_BF16 ? launch_typed<__nv_bfloat16>(p, stream)
                            : launch_typed<float>(p, stream);
}

}  // namespace dard
