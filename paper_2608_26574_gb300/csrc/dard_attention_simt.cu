// dard_attention_simt.cu - the fp32 attention kernel on CUDA cores (dtype F32): the
// validation path and the kernel of fp32 workloads. Same mask as the tensor-core kernels
// (Sec. 3.1 Eq. 2; Sec. 3.2 query blocks 1-6, Eq. 3), through key_visible(), and the same
// RoPE positions (dard_rope.cuh).
#include "dard_attn_common.cuh"

namespace dard {
namespace {

// ---------------------------------------------------------------- fp32 CUDA-core path
// A CTA holds 32 query rows of one head (a quarter of a 128-row query tile), four threads per
// row in each of four key groups, 512 threads: thread `part` of a row owns the four-element
// vectors 16 v + 4 part .. 16 v + 4 part + 3 (v = 0 .. D/16 - 1) of q and of its O
// accumulator, so that the row's four threads read 64 contiguous bytes of a shared-memory
// key row per vector (one 16-byte load each, no bank conflict). The sequence's keys pass
// through shared memory 32 rows at a time (K and V, read as broadcasts; each thread loads
// its share of the next tile while the current one is computed); key group `grp` takes
// keys 8 grp .. 8 grp + 7 of every tile, four at a time: four independent partial dot
// products, which the row's four threads add up with two shuffles each, then one online
// softmax step over the four. At the end the four groups' (maximum, sum, accumulator) of a
// row are merged through shared memory. Masking as on the tensor-core path, by
// key_visible().
constexpr int kSimtRows = 32;     // query rows per CTA
constexpr int kSimtParts = 4;     // threads per query row and key group
constexpr int kSimtGroups = 4;    // key groups
constexpr int kSimtGroupThreads = kSimtRows * kSimtParts;
constexpr int kSimtThreads = kSimtGroupThreads * kSimtGroups;
constexpr int kSimtSplit = kSimtCtasPerTile;  // CTAs per 128-row query tile
static_assert(kSimtSplit * kSimtRows == kBM, "the CTAs cover a 128-row query tile");

template <int D>
__global__ void __launch_bounds__(kSimtThreads) attn_simt(const __grid_constant__ AttnParams p) {
  constexpr int kV = D / 16;                   // float4 vectors per thread
  constexpr int kKT = 32;                      // keys per shared-memory tile
  constexpr int kKG = kKT / kSimtGroups;       // keys of a tile per key group
  static_assert(kKG % 4 == 0, "four keys per step");
  static_assert(kKT >= kSimtRows, "the merge reuses the K and V tile buffers, one row block each");
  __shared__ BlockInfo bi;
  __shared__ __align__(16) float sK[kKT][D];
  __shared__ __align__(16) float sV[kKT][D];
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
  // vector v of this thread: float4 index 4 v + part of the row
  const size_t qoff4 = (static_cast<size_t>(sd.row_base + r) * p.hq + h) * (D / 4) + part;
  float4 qv[kV], acc[kV];
#pragma unroll
  for (int v = 0; v < kV; ++v) {
    qv[v] = live ? reinterpret_cast<const float4*>(Q)[qoff4 + 4 * v] : make_float4(0.f, 0.f, 0.f, 0.f);
    acc[v] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  if (p.rope && live) {  // RoPE of this row; its pairs lie within one thread
    const int pos = rope_position(p, sd, r);
    auto rot = [](float& a, float& b, float c, float s) {
      const float x = a, y = b;
      a = fmaf(x, c, -y * s);
      b = fmaf(x, s, y * c);
    };
    if (p.rope_style == DARD_ROPE_INTERLEAVED) {
      // elements (d, d + 1) of a vector, d = 16 v + 4 part + {0, 2}: frequency d / 2
#pragma unroll
      for (int v = 0; v < kV; ++v) {
        const int i = 8 * v + 2 * part;
        float c0, s0, c1, s1;
        rope_cos_sin(pos, p.rope_f[2 * i], p.rope_f[2 * i + 1], c0, s0);
        rope_cos_sin(pos, p.rope_f[2 * i + 2], p.rope_f[2 * i + 3], c1, s1);
        rot(qv[v].x, qv[v].y, c0, s0);
        rot(qv[v].z, qv[v].w, c1, s1);
      }
    } else {
      // element d = 16 v + 4 part + k < D/2 pairs with d + D/2 (vector v + kV/2): frequency d
#pragma unroll
      for (int v = 0; v < kV / 2; ++v) {
        const int i = 16 * v + 4 * part;
        float c[4], s[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) rope_cos_sin(pos, p.rope_f[2 * (i + k)], p.rope_f[2 * (i + k) + 1], c[k], s[k]);
        float4& a = qv[v];
        float4& b = qv[v + kV / 2];
        rot(a.x, b.x, c[0], s[0]);
        rot(a.y, b.y, c[1], s[1]);
        rot(a.z, b.z, c[2], s[2]);
        rot(a.w, b.w, c[3], s[3]);
      }
    }
  }
  grid_dep_wait();  // the RoPE key pass launched before this kernel (if any) is complete
  // K/V tiles are software-pipelined: each thread holds its share of the next tile in
  // registers, loaded while the current tile is computed
  constexpr int kLoads = kKT * D / 4 / kSimtThreads;  // float4 of K (and of V) per thread
  static_assert(kKT * D / 4 % kSimtThreads == 0, "a tile splits evenly over the threads");
  float4 nxk[kLoads], nxv[kLoads];
  auto fetch = [&](int kt0) {
#pragma unroll
    for (int u = 0; u < kLoads; ++u) {
      const int idx = static_cast<int>(threadIdx.x) + u * kSimtThreads;
      const int kr = kt0 + idx / (D / 4), c4 = idx % (D / 4);
      nxk[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      nxv[u] = nxk[u];
      if (kr < rows_seq) {
        const size_t off = (static_cast<size_t>(sd.row_base + kr) * p.hkv + g) * (D / 4) + c4;
        nxk[u] = reinterpret_cast<const float4*>(K)[off];
        nxv[u] = reinterpret_cast<const float4*>(V)[off];
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
      reinterpret_cast<float4*>(sK[idx / (D / 4)])[idx % (D / 4)] = nxk[u];
      reinterpret_cast<float4*>(sV[idx / (D / 4)])[idx % (D / 4)] = nxv[u];
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
      for (int v = 0; v < kV; ++v) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float4 kx = reinterpret_cast<const float4*>(sK[kk + u])[4 * v + part];
          dot[u] = fmaf(qv[v].x, kx.x, dot[u]);
          dot[u] = fmaf(qv[v].y, kx.y, dot[u]);
          dot[u] = fmaf(qv[v].z, kx.z, dot[u]);
          dot[u] = fmaf(qv[v].w, kx.w, dot[u]);
        }
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
        for (int v = 0; v < kV; ++v) {
          acc[v].x *= alpha;
          acc[v].y *= alpha;
          acc[v].z *= alpha;
          acc[v].w *= alpha;
        }
        m = zmax;
      }
      float pz[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        pz[u] = vis[u] ? expf(z[u] - m) : 0.f;
        l += pz[u];
      }
#pragma unroll
      for (int v = 0; v < kV; ++v) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float4 vx = reinterpret_cast<const float4*>(sV[kk + u])[4 * v + part];
          acc[v].x = fmaf(pz[u], vx.x, acc[v].x);
          acc[v].y = fmaf(pz[u], vx.y, acc[v].y);
          acc[v].z = fmaf(pz[u], vx.z, acc[v].z);
          acc[v].w = fmaf(pz[u], vx.w, acc[v].w);
        }
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
      float4* slot = reinterpret_cast<float4*>(grp == half ? &sK[0][0] : &sV[0][0]);
#pragma unroll
      for (int v = 0; v < kV; ++v) slot[t * (D / 4) + 4 * v + part] = acc[v];
    }
    __syncthreads();
    if (grp < half) {
      const float4* slot = reinterpret_cast<const float4*>(grp == 0 ? &sK[0][0] : &sV[0][0]);
      const float mo = s_m[grp + half][t], lo = s_l[grp + half][t];
      const float mn = fmaxf(m, mo);
      const float a = (m == -INFINITY) ? 0.f : expf(m - mn);
      const float b = (mo == -INFINITY) ? 0.f : expf(mo - mn);
      l = l * a + lo * b;
#pragma unroll
      for (int v = 0; v < kV; ++v) {
        const float4 o = slot[t * (D / 4) + 4 * v + part];
        acc[v].x = acc[v].x * a + o.x * b;
        acc[v].y = acc[v].y * a + o.y * b;
        acc[v].z = acc[v].z * a + o.z * b;
        acc[v].w = acc[v].w * a + o.w * b;
      }
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
    for (int v = 0; v < kV; ++v)
      reinterpret_cast<float4*>(O)[qoff4 + 4 * v] =
          make_float4(acc[v].x * inv_l, acc[v].y * inv_l, acc[v].z * inv_l, acc[v].w * inv_l);
  }
}

}  // namespace

cudaError_t launch_simt_attention(const AttnParams& p, cudaStream_t stream) {
  const AttnLaunch L(p.total_work * kSimtSplit, kSimtThreads, 0, stream, 1, p.rope != 0);
  return p.head_dim == 64 ? cudaLaunchKernelEx(&L.cfg, attn_simt<64>, p)
                          : cudaLaunchKernelEx(&L.cfg, attn_simt<128>, p);
}

}  // namespace dard
