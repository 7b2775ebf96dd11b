// Prefill cache fill (Sec. 5, "Chunked-Prefill Stage"): a chunk of rows at
// positions Lb .. Lb + len - 1 is appended after Lb cached tokens. Retrieval
// KV heads keep every position; streaming KV heads keep the S sinks and the
// last W positions of the new length, position p >= S going to ring row
// S + (p - S) mod W (overwriting the positions that leave the window).
//
// One CTA copies ROWS token rows of one (sequence, KV head) for K and V.
// Each row is D bf16 = D/8 16-byte chunks; consecutive threads take
// consecutive chunks, so loads and stores are coalesced 16-byte accesses.
#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

using bf16 = __nv_bfloat16;
constexpr int kRows = 64;
constexpr int kThreads = 256;

template <int D>
__global__ void __launch_bounds__(kThreads) append_kernel(const __grid_constant__ AppendArgs a) {
  constexpr int CPR = D / 8;  // 16-byte chunks per row
  constexpr int RPI = kThreads / CPR;
  const CacheGeom& g = a.geom;
  const int b = blockIdx.z, h = blockIdx.y;
  const int len = a.lens[b];
  const int Lb = a.base[b];
  const int newlen = Lb + len;
  const int r0 = blockIdx.x * kRows;          // chunk rows [r0, r1)
  const int r1 = min(r0 + kRows, len);
  if (r0 >= r1) return;
  const bool streaming = g.kind[h] != 0;
  if (streaming && Lb + r1 <= newlen - g.W && Lb + r0 >= g.S) return;  // rows neither sink nor window
  const int cap = g.capacity(h);
  uint4* Kd = reinterpret_cast<uint4*>(static_cast<bf16*>(a.kv) + g.region(b, h));
  uint4* Vd = Kd + (size_t)cap * CPR;
  const uint4* Ks = static_cast<const uint4*>(a.k);
  const uint4* Vs = static_cast<const uint4*>(a.v);
  const int ch = threadIdx.x % CPR;
  for (int r = r0 + threadIdx.x / CPR; r < r1; r += RPI) {
    const int p = Lb + r;
    int dst = p;
    if (streaming && p >= g.S) {
      if (p < newlen - g.W) continue;
      dst = g.S + (p - g.S) % g.W;
    }
    const size_t src = (((size_t)b * a.T + r) * g.Hkv + h) * CPR + ch;
    Kd[(size_t)dst * CPR + ch] = Ks[src];
    Vd[(size_t)dst * CPR + ch] = Vs[src];
  }
}

// lens[b] += add[b] (the lengths after a prefill chunk), stream-ordered.
__global__ void lens_add_kernel(int32_t* lens, const int32_t* add, int B) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) lens[b] += add[b];
}

}  // namespace

cudaError_t launch_lens_add(int32_t* lens, const int32_t* add, int B, cudaStream_t s) {
  lens_add_kernel<<<(B + 255) / 256, 256, 0, s>>>(lens, add, B);
  return cudaGetLastError();
}

cudaError_t launch_append(const AppendArgs& a, cudaStream_t s) {
  dim3 grid((a.T + kRows - 1) / kRows, a.geom.Hkv, a.geom.B);
  if (a.geom.D == 128)
    append_kernel<128><<<grid, kThreads, 0, s>>>(a);
  else if (a.geom.D == 64)
    append_kernel<64><<<grid, kThreads, 0, s>>>(a);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace aoh
