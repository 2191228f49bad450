// dard_attention_simt.cu - the fp32 attention kernel on CUDA cores (dtype F32): the
// validation path and the kernel of fp32 workloads. Same mask as the tensor-core kernels
// (Sec. 3.1 Eq. 2; Sec. 3.2 query blocks 1-6, Eq. 3), through key_visible(), and the same
// RoPE positions (dard_rope.cuh).
#include "dard_attn_common.cuh"

namespace dard {
namespace {

// ---------------------------------------------------------------- fp32 CUDA-core path
// A CTA holds 32 query rows of one head (a quarter of a 128-row query tile), four threads per
// row in each of four key groups, 512 threads: thread `part` of a row owns elements part,
// part + 4, ... of q and of its O accumulator. The sequence's keys pass through shared
// memory 32 rows at a time (K and V, read as broadcasts); key group `grp` takes keys
// 8 grp .. 8 grp + 7 of every tile, four at a time: four independent partial dot products,
// which the row's four threads add up with two shuffles each, then one online softmax step
// over the four. At the end the four groups' (maximum, sum, accumulator) of a row are
// merged through shared memory. Masking as on the tensor-core path, by key_visible().
constexpr int kSimtRows = 32;     // query rows per CTA
constexpr int kSimtParts = 4;     // threads per query row and key group
constexpr int kSimtGroups = 4;    // key groups
constexpr int kSimtGroupThreads = kSimtRows * kSimtParts;
constexpr int kSimtThreads = kSimtGroupThreads * kSimtGroups;
constexpr int kSimtSplit = kSimtCtasPerTile;  // CTAs per 128-row query tile
static_assert(kSimtSplit * kSimtRows == kBM, "the CTAs cover a 128-row query tile");

template <int D>
__global__ void __launch_bounds__(kSimtThreads) attn_simt(const __grid_constant__ AttnParams p) {
  constexpr int kE = D / kSimtParts;           // elements per thread
  constexpr int kKT = 32;                      // keys per shared-memory tile
  constexpr int kKG = kKT / kSimtGroups;       // keys of a tile per key group
  static_assert(kKG % 4 == 0, "four keys per step");
  static_assert(kKT >= kSimtRows, "the merge reuses the K and V tile buffers, one row block each");
  __shared__ BlockInfo bi;
  __shared__ float sK[kKT][D], sV[kKT][D];
  __shared__ float s_m[kSimtGroups][kSimtRows], s_l[kSimtGroups][kSimtRows];
  int seq, qt, h;
  decode_work(p, blockIdx.x / kSimtSplit, seq, qt, h);
  const int sub = blockIdx.x % kSimtSplit;
  const SeqDesc sd = p.seq[seq];
  const int rows_seq = sd.n_orig + sd.slen;
  const int g = h / (p.hq / p.hkv);
  if (threadIdx.x < 128)  // warps 0-3
    load_block_info(p, sd, bi, qt == 0 && h == 0 && sub == 0);
  __syncthreads();
  const int grp = threadIdx.x / kSimtGroupThreads, local = threadIdx.x % kSimtGroupThreads;
  const int t = local / kSimtParts, part = local % kSimtParts;
  const unsigned quad = 0xfu << ((threadIdx.x & 31) & ~3);  // the row's four threads
  const int r = sd.q_start + qt * kBM + sub * kSimtRows + t;  // sequence-relative query row
  const bool active = r < rows_seq;
  RowInfo q{0, kStateU, 0.f, -1, 0};
  if (active) q = row_info(sd, bi, r);
  const bool live = active && q.store;
  const float* Q = static_cast<const float*>(p.q);
  const float* K = static_cast<const float*>(p.k);
  const float* V = static_cast<const float*>(p.v);
  float* O = static_cast<float*>(p.o);
  const size_t qoff = (static_cast<size_t>(sd.row_base + r) * p.hq + h) * D + part;
  float qv[kE], acc[kE];
#pragma unroll
  for (int e = 0; e < kE; ++e) {
    qv[e] = live ? Q[qoff + kSimtParts * e] : 0.f;
    acc[e] = 0.f;
  }
  if (p.rope && live) {  // RoPE of this row; the row's four threads take this branch together
    const int pos = rope_position(p, sd, r);
    if (p.rope_style == DARD_ROPE_INTERLEAVED) {
      // element 4e + part pairs with 4e + (part ^ 1), frequency 2e + part / 2
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        const int i = 2 * e + part / 2;
        float c, s;
        rope_cos_sin(pos, p.rope_f[2 * i], p.rope_f[2 * i + 1], c, s);
        const float other = __shfl_xor_sync(quad, qv[e], 1);
        qv[e] = (part & 1) == 0 ? fmaf(qv[e], c, -other * s) : fmaf(other, s, qv[e] * c);
      }
    } else {
      // element d = 4e + part < D/2 pairs with d + D/2 = 4 (e + D/8) + part, frequency d
#pragma unroll
      for (int e = 0; e < kE / 2; ++e) {
        const int i = kSimtParts * e + part;
        float c, s;
        rope_cos_sin(pos, p.rope_f[2 * i], p.rope_f[2 * i + 1], c, s);
        const float a = qv[e], b = qv[e + kE / 2];
        qv[e] = fmaf(a, c, -b * s);
        qv[e + kE / 2] = fmaf(a, s, b * c);
      }
    }
  }
  grid_dep_wait();  // the RoPE key pass launched before this kernel (if any) is complete
  // K/V tiles are software-pipelined: each thread holds its share of the next tile in
  // registers, loaded while the current tile is computed
  constexpr int kLoads = kKT * D / kSimtThreads;  // elements of K (and of V) per thread
  static_assert(kKT * D % kSimtThreads == 0, "a tile splits evenly over the threads");
  float nxk[kLoads], nxv[kLoads];
  auto fetch = [&](int kt0) {
#pragma unroll
    for (int u = 0; u < kLoads; ++u) {
      const int idx = static_cast<int>(threadIdx.x) + u * kSimtThreads;
      const int kr = kt0 + idx / D, d = idx % D;
      nxk[u] = 0.f;
      nxv[u] = 0.f;
      if (kr < rows_seq) {
        const size_t off = (static_cast<size_t>(sd.row_base + kr) * p.hkv + g) * D + d;
        nxk[u] = K[off];
        nxv[u] = V[off];
      }
    }
  };
  fetch(0);
  float m = -INFINITY, l = 0.f;
  for (int kt0 = 0; kt0 < rows_seq; kt0 += kKT) {
    __syncthreads();  // the previous tile has been read
#pragma unroll
    for (int u = 0; u < kLoads; ++u) {
      const int idx = static_cast<int>(threadIdx.x) + u * kSimtThreads;
      sK[idx / D][idx % D] = nxk[u];
      sV[idx / D][idx % D] = nxv[u];
    }
    __syncthreads();
    if (kt0 + kKT < rows_seq) fetch(kt0 + kKT);
    if (!live) continue;
    const int k_end = min(kKT, rows_seq - kt0);
    // four keys per step: four independent dot-product chains, one maximum and at most one
    // rescale per step (keys past the sequence or hidden by the mask weigh 0)
    for (int kk = grp * kKG; kk < grp * kKG + kKG && kk < k_end; kk += 4) {
      bool vis[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        vis[u] = kk + u < k_end && key_visible(q, bi, sd, kt0 + kk + u);  // the same for the row
      if (!(vis[0] || vis[1] || vis[2] || vis[3])) continue;
      float dot[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int e = 0; e < kE; ++e) {
#pragma unroll
        for (int u = 0; u < 4; ++u) dot[u] = fmaf(qv[e], sK[kk + u][kSimtParts * e + part], dot[u]);
      }
      float z[4];
      float zmax = -INFINITY;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        dot[u] += __shfl_xor_sync(quad, dot[u], 1);
        dot[u] += __shfl_xor_sync(quad, dot[u], 2);
        z[u] = vis[u] ? dot[u] * p.scale : -INFINITY;
        zmax = fmaxf(zmax, z[u]);
      }
      if (zmax > m) {
        const float alpha = (m == -INFINITY) ? 0.f : expf(m - zmax);
        l *= alpha;
#pragma unroll
        for (int e = 0; e < kE; ++e) acc[e] *= alpha;
        m = zmax;
      }
      float pz[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        pz[u] = vis[u] ? expf(z[u] - m) : 0.f;
        l += pz[u];
      }
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        float a = acc[e];
#pragma unroll
        for (int u = 0; u < 4; ++u) a = fmaf(pz[u], sV[kk + u][kSimtParts * e + part], a);
        acc[e] = a;
      }
    }
  }
  // Merge the key groups: groups 2 and 3 hand their state to groups 0 and 1, then group 1
  // to group 0, through the K and V tile buffers (free once every group is past its last
  // tile): group half + k writes into buffer k (sK for k = 0, sV for k = 1).
  if (part == 0) {
    s_m[grp][t] = m;
    s_l[grp][t] = l;
  }
  __syncthreads();
#pragma unroll
  for (int half = 2; half >= 1; half >>= 1) {
    if (grp >= half && grp < 2 * half) {
      float* slot = grp == half ? &sK[0][0] : &sV[0][0];
#pragma unroll
      for (int e = 0; e < kE; ++e) slot[t * D + kSimtParts * e + part] = acc[e];
    }
    __syncthreads();
    if (grp < half) {
      const float* slot = grp == 0 ? &sK[0][0] : &sV[0][0];
      const float mo = s_m[grp + half][t], lo = s_l[grp + half][t];
      const float mn = fmaxf(m, mo);
      const float a = (m == -INFINITY) ? 0.f : expf(m - mn);
      const float b = (mo == -INFINITY) ? 0.f : expf(mo - mn);
      l = l * a + lo * b;
#pragma unroll
      for (int e = 0; e < kE; ++e)
        acc[e] = acc[e] * a + slot[t * D + kSimtParts * e + part] * b;
      m = mn;
    }
    __syncthreads();
    if (grp < half && part == 0) {
      s_m[grp][t] = m;
      s_l[grp][t] = l;
    }
    __syncthreads();
  }
  if (live && grp == 0) {
    const float inv_l = 1.0f / l;
#pragma unroll
    for (int e = 0; e < kE; ++e) O[qoff + kSimtParts * e] = acc[e] * inv_l;
  }
}

}  // namespace

cudaError_t launch_simt_attention(const AttnParams& p, cudaStream_t stream) {
  const AttnLaunch L(p.total_work * kSimtSplit, kSimtThreads, 0, stream, 1, p.rope != 0);
  return p.head_dim == 64 ? cudaLaunchKernelEx(&L.cfg, attn_simt<64>, p)
                          : cudaLaunchKernelEx(&L.cfg, attn_simt<128>, p);
}

}  // namespace dard
