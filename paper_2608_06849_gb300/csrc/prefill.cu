// Causal prefill attention with retrieval / streaming masks (Sec. 5,
// "Chunked-Prefill Stage", with the per-token sink + window rule).
//
// First correct version on CUDA cores: one CTA = 64 query rows of one query
// head, two threads per row (each owns half of d_head). K/V tiles of 64 keys
// are staged in shared memory; only tiles that intersect the visible set are
// visited (for a streaming head: the sink tiles and the window tiles).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

using bf16 = __nv_bfloat16;
constexpr int kQT = 64, kKT = 64, kChunk = 16;

template <int D>
__global__ void __launch_bounds__(128) prefill_simple_kernel(const __grid_constant__ PrefillArgs a) {
  constexpr int H2 = D / 2;
  __shared__ __align__(16) bf16 Ks[kKT][D];
  __shared__ __align__(16) bf16 Vs[kKT][D];
  const CacheGeom& g = a.geom;
  const int b = blockIdx.z, h = blockIdx.y, kvh = h / g.G;
  const int len = a.lens[b];
  const int q0 = blockIdx.x * kQT;
  if (q0 >= len) return;
  const int row = threadIdx.x >> 1, half = threadIdx.x & 1;
  const int i = q0 + row;
  const bool streaming = g.kind[kvh] != 0;
  const int S = g.S, W = g.W;

  float q[H2], o[H2];
  const bf16* qp = static_cast<const bf16*>(a.q) + (((size_t)b * a.T + min(i, len - 1)) * g.Hq + h) * D + half * H2;
#pragma unroll
  for (int e = 0; e < H2; e += 2) {
    const float2 f = bf16x2_to_float2(*reinterpret_cast<const uint32_t*>(qp + e));
    q[e] = f.x * a.scale_log2;
    q[e + 1] = f.y * a.scale_log2;
    o[e] = o[e + 1] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  const int q_end = min(q0 + kQT, len);

  for (int j0 = 0; j0 < q_end; j0 += kKT) {
    if (streaming) {
      const bool in_sink = j0 < S;
      const bool in_window = j0 + kKT - 1 > q0 - W;  // some key j with q_end-1 - j < W ... conservative
      if (!in_sink && !in_window) continue;
    }
    __syncthreads();
    for (int x = threadIdx.x; x < kKT * D / 8; x += blockDim.x) {
      const int r = x / (D / 8), ch = x % (D / 8);
      const int j = min(j0 + r, len - 1);
      const size_t src = (((size_t)b * a.T + j) * g.Hkv + kvh) * D + ch * 8;
      *reinterpret_cast<uint4*>(&Ks[r][ch * 8]) = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(a.k) + src);
      *reinterpret_cast<uint4*>(&Vs[r][ch * 8]) = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(a.v) + src);
    }
    __syncthreads();
    for (int c0 = 0; c0 < kKT; c0 += kChunk) {
      float s[kChunk];
      float cmax = -INFINITY;
#pragma unroll
      for (int jj = 0; jj < kChunk; ++jj) {
        const bf16* kr = &Ks[c0 + jj][half * H2];
        float acc = 0.f;
#pragma unroll
        for (int e = 0; e < H2; e += 2) {
          const float2 f = bf16x2_to_float2(*reinterpret_cast<const uint32_t*>(kr + e));
          acc = fmaf(q[e], f.x, acc);
          acc = fmaf(q[e + 1], f.y, acc);
        }
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        const int j = j0 + c0 + jj;
        const bool ok = (j <= i) && (j < len) && (!streaming || j < S || i - j < W);
        s[jj] = ok ? acc : -INFINITY;
        cmax = fmaxf(cmax, s[jj]);
      }
      const float mn = fmaxf(m, cmax);
      if (mn == -INFINITY) continue;
      const float alpha = (m == -INFINITY) ? 0.f : fast_exp2(m - mn);
      m = mn;
      l *= alpha;
#pragma unroll
      for (int e = 0; e < H2; ++e) o[e] *= alpha;
#pragma unroll
      for (int jj = 0; jj < kChunk; ++jj) {
        const float p = (s[jj] == -INFINITY) ? 0.f : fast_exp2(s[jj] - m);
        l += p;
        const bf16* vr = &Vs[c0 + jj][half * H2];
#pragma unroll
        for (int e = 0; e < H2; e += 2) {
          const float2 f = bf16x2_to_float2(*reinterpret_cast<const uint32_t*>(vr + e));
          o[e] = fmaf(p, f.x, o[e]);
          o[e + 1] = fmaf(p, f.y, o[e + 1]);
        }
      }
    }
  }
  if (i < len && a.out != nullptr) {
    bf16* op = static_cast<bf16*>(a.out) + (((size_t)b * a.T + i) * g.Hq + h) * D + half * H2;
    const float inv = 1.f / l;
#pragma unroll
    for (int e = 0; e < H2; e += 2)
      *reinterpret_cast<uint32_t*>(op + e) = float2_to_bf16x2(o[e] * inv, o[e + 1] * inv);
  }
}

}  // namespace

bool prefill_supported(int D, int G) { return (D == 64 || D == 128) && G >= 1; }

cudaError_t launch_prefill(const PrefillArgs& a, cudaStream_t s) {
  dim3 grid((a.T + kQT - 1) / kQT, a.geom.Hq, a.geom.B);
  if (a.geom.D == 128)
    prefill_simple_kernel<128><<<grid, 128, 0, s>>>(a);
  else if (a.geom.D == 64)
    prefill_simple_kernel<64><<<grid, 128, 0, s>>>(a);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace aoh
