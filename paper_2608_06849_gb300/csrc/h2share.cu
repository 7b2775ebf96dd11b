// H2Share anchor-layer selection (the paper's H2Share section and its GQA
// extension appendix): after an anchor decode step that wrote the scores of
// every retrieval row, each (sequence, retrieval KV head) keeps the top_k
// positions by group importance, the sum over the group's query heads of
// their attention probabilities. Ties go to the lower position; the
// positions are listed in increasing order, padded with -1 when fewer than
// top_k rows are held.
//
// The decode kernel leaves each retrieval head's final softmax state
// (M_h, L_h = sum of 2^(s - M_h), log2 units) beside the scores. Then:
//   h2_imp_kernel     over (row chunk, item), so the whole GPU streams the
//                     scores: importance_j = sum_h 2^(s_hj - M_h) / L_h,
//                     written once,
//                     and counts the top 11 bits of every importance into the
//                     item's histogram (importance is >= 0, so its bit
//                     pattern orders like its value; the select kernel
//                     zeroes the histogram again after reading it);
//   h2_select_kernel  one CTA per item: the histogram bucket that holds the
//                     top_k-th largest value, the exact threshold among that
//                     bucket's members (gathered into shared memory; full
//                     radix passes over the item when the bucket is too
//                     large), then an ordered compaction: each warp owns a
//                     contiguous run of rows and walks it 32 rows at a time;
//                     a scan over the warps and ballots within them place
//                     the rows above the threshold and, in position order,
//                     as many rows equal to it as the rank still needs.
#include <stdint.h>

#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

constexpr int kChunk = 8192;          // rows per chunk of the importance kernel
constexpr int kChunkThreads = 256;
constexpr int kSelThreads = 1024;
constexpr int kBins = 2048;           // top 11 bits
constexpr int kCand = 8192;           // candidates kept in shared memory

template <int G>
__global__ void __launch_bounds__(kChunkThreads) h2_imp_kernel(const float* scores, int stride, const int32_t* lens,
                                                               int n_r, const float2* stats, float* imp_all,
                                                               uint32_t* hist) {
  __shared__ float Mh[16], Linv[16];
  __shared__ uint32_t sh_hist[kBins];
  const int chunk = blockIdx.x, item = blockIdx.y, b = item / n_r;
  const int n = __ldcg(&lens[b]);
  if (threadIdx.x < G) {
    const float2 st = __ldcg(&stats[(size_t)item * G + threadIdx.x]);
    Mh[threadIdx.x] = st.x;
    Linv[threadIdx.x] = 1.f / st.y;
  }
  for (int i = threadIdx.x; i < kBins; i += kChunkThreads) sh_hist[i] = 0u;
  __syncthreads();
  const int j0 = chunk * kChunk, j1 = min(n, j0 + kChunk);
  float* imp = imp_all + (size_t)item * stride;
  // U rows per thread and step, every score load of the step issued before
  // any is used (the histogram atomics would otherwise keep the next row's
  // loads from being hoisted, leaving G loads in flight per thread)
  constexpr int U = 4;
  for (int jb = j0; jb < j1; jb += U * kChunkThreads) {
    float sv[U][G];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * kChunkThreads + threadIdx.x;
#pragma unroll
      for (int h = 0; h < G; ++h) sv[u][h] = j < j1 ? __ldcg(scores + ((size_t)item * G + h) * stride + j) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * kChunkThreads + threadIdx.x;
      float v = 0.f;
#pragma unroll
      for (int h = 0; h < G; ++h) v += fast_exp2(sv[u][h] - Mh[h]) * Linv[h];
      if (j < j1) imp[j] = v;
      // warp-aggregated: most importances are tiny and share a few bins
      const uint32_t bin = j < j1 ? __float_as_uint(v) >> 21 : 0xffffffffu;
      const unsigned peers = __match_any_sync(0xffffffffu, bin);
      if (j < j1 && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&sh_hist[bin], (uint32_t)__popc(peers));
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kBins; i += kChunkThreads)
    if (sh_hist[i]) atomicAdd(&hist[(size_t)item * kBins + i], sh_hist[i]);
}

// Exclusive block scan of one int per thread (kSelThreads); ws holds 32 ints.
__device__ int block_exclusive_scan(int v, int* ws) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  __syncthreads();
  if (lane == 31) ws[warp] = inc;
  __syncthreads();
  if (threadIdx.x == 0) {
    int run = 0;
    for (int w = 0; w < kSelThreads / 32; ++w) {
      const int x = ws[w];
      ws[w] = run;
      run += x;
    }
  }
  __syncthreads();
  return ws[warp] + inc - v;
}

// Among values whose bits match `prefix` under `mask`, the bucket of digit
// (bits >> shift) & (nb - 1), counted from the top, that holds the rank-th
// largest; returns the digit and leaves the rank within it in *rank.
__device__ uint32_t top_bucket(const uint32_t* h, int nb, int* rank, int* ws) {
  const int per = nb / kSelThreads;  // nb (2048) is a multiple of kSelThreads
  // thread t covers digits nb-1-t*per .. nb-per-t*per (from the top)
  int mine = 0;
  for (int i = 0; i < per; ++i) mine += (int)h[nb - 1 - threadIdx.x * per - i];
  const int before = block_exclusive_scan(mine, ws);
  __shared__ uint32_t sh_digit;
  __shared__ int sh_rank;
  const int r = *rank;
  if (before < r && before + mine >= r) {
    int acc = before;
    for (int i = 0; i < per; ++i) {
      const uint32_t d = nb - 1 - threadIdx.x * per - i;
      if (acc + (int)h[d] >= r) {
        sh_digit = d;
        sh_rank = r - acc;
        break;
      }
      acc += h[d];
    }
  }
  __syncthreads();
  *rank = sh_rank;
  return sh_digit;
}

__global__ void __launch_bounds__(kSelThreads) h2_select_kernel(const int32_t* lens, int n_r, int stride, int top_k,
                                                                const float* imp_all, uint32_t* hist_all,
                                                                int32_t* idx_all) {
  __shared__ int ws[32];
  __shared__ uint32_t h2[kBins];
  __shared__ uint32_t cand[kCand];
  __shared__ int n_cand;
  const int item = blockIdx.x, b = item / n_r;
  const int n = __ldcg(&lens[b]);
  const float* imp = imp_all + (size_t)item * stride;
  int32_t* out = idx_all + (size_t)item * top_k;
  uint32_t* hist = hist_all + (size_t)item * kBins;
  if (n <= top_k) {
    for (int j = threadIdx.x; j < top_k; j += kSelThreads) out[j] = j < n ? j : -1;
    // the importance kernel counted this step's rows: zero them for the next
    for (int i = threadIdx.x; i < kBins; i += kSelThreads) hist[i] = 0u;
    return;
  }
  for (int i = threadIdx.x; i < kBins; i += kSelThreads) {
    h2[i] = __ldcg(hist + i);
    hist[i] = 0u;  // zero again for the next step
  }
  if (threadIdx.x == 0) n_cand = 0;
  __syncthreads();
  int rank = top_k;
  const uint32_t d1 = top_bucket(h2, kBins, &rank, ws);  // bits 31..21
  // gather the bucket's members (one shared atomic per warp and step)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned below = (1u << lane) - 1u;
  constexpr int U = 8;  // steps whose loads are issued together
  for (int jb = 0; jb < n; jb += kSelThreads * U) {
    uint32_t v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * kSelThreads + threadIdx.x;
      v[u] = j < n ? __float_as_uint(__ldcg(imp + j)) : 0u;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * kSelThreads + threadIdx.x;
      const bool member = j < n && (v[u] >> 21) == d1;
      const unsigned mm = __ballot_sync(0xffffffffu, member);
      if (mm) {
        int base = 0;
        if (lane == __ffs(mm) - 1) base = atomicAdd(&n_cand, __popc(mm));
        base = __shfl_sync(0xffffffffu, base, __ffs(mm) - 1);
        const int c = base + __popc(mm & below);
        if (member && c < kCand) cand[c] = v[u];
      }
    }
  }
  __syncthreads();
  const int nc = n_cand;
  // digits 20..10 (11 bits) and 9..0 (10 bits) of the threshold
  uint32_t prefix = d1 << 21, mask = 0xFFE00000u;
  const int shifts[2] = {10, 0};
  const int widths[2] = {11, 10};
  for (int level = 0; level < 2; ++level) {
    const int sh = shifts[level], nb = 1 << widths[level];
    for (int i = threadIdx.x; i < kBins; i += kSelThreads) h2[i] = 0u;
    __syncthreads();
    if (nc <= kCand) {
      for (int c = threadIdx.x; c < nc; c += kSelThreads)
        if ((cand[c] & mask) == prefix) atomicAdd(&h2[(cand[c] >> sh) & (nb - 1)], 1u);
    } else {
      for (int j = threadIdx.x; j < n; j += kSelThreads) {
        const uint32_t bits = __float_as_uint(__ldcg(imp + j));
        if ((bits & mask) == prefix) atomicAdd(&h2[(bits >> sh) & (nb - 1)], 1u);
      }
    }
    __syncthreads();
    const uint32_t d = top_bucket(h2, kBins, &rank, ws);  // digits above nb - 1 are empty
    prefix |= d << sh;
    mask |= (uint32_t)(nb - 1) << sh;
    __syncthreads();
  }
  const uint32_t thr = prefix;
  const int need_eq = rank;
  // ordered compaction: warp w owns rows [w*seg, (w+1)*seg) and walks them
  // 32 at a time (coalesced); ballots give every selected row its place
  constexpr int kWarps = kSelThreads / 32;
  const int seg = (n + kWarps - 1) / kWarps;
  const int w0 = min(n, warp * seg), w1 = min(n, w0 + seg);
  int gt = 0, eq = 0;
  for (int jb = w0; jb < w1; jb += 32 * U) {
    uint32_t v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * 32 + lane;
      v[u] = j < w1 ? __float_as_uint(__ldcg(imp + j)) : 0u;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const bool in = jb + u * 32 + lane < w1;
      gt += in && v[u] > thr;
      eq += in && v[u] == thr;
    }
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    gt += __shfl_xor_sync(0xffffffffu, gt, o);
    eq += __shfl_xor_sync(0xffffffffu, eq, o);
  }
  // per-warp counts -> exclusive prefixes over warps (lane 0 of each warp
  // holds the counts; the scan runs over threads, non-leaders add zero)
  const int eq_before = block_exclusive_scan(lane == 0 ? eq : 0, ws);
  const int take_eq = max(0, min(eq, need_eq - __shfl_sync(0xffffffffu, eq_before, 0)));
  const int pos0 = block_exclusive_scan(lane == 0 ? gt + take_eq : 0, ws);
  int pos = __shfl_sync(0xffffffffu, pos0, 0);
  int taken = 0;  // equal rows taken so far by this warp
  for (int jb = w0; jb < w1; jb += 32 * U) {
    uint32_t v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * 32 + lane;
      v[u] = j < w1 ? __float_as_uint(__ldcg(imp + j)) : 0u;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int j = jb + u * 32 + lane;
      const bool is_gt = j < w1 && v[u] > thr;
      const bool is_eq = j < w1 && v[u] == thr;
      const unsigned eqm = __ballot_sync(0xffffffffu, is_eq);
      const bool keep = is_gt || (is_eq && taken + __popc(eqm & below) < take_eq);
      const unsigned km = __ballot_sync(0xffffffffu, keep);
      if (keep) out[pos + __popc(km & below)] = j;
      pos += __popc(km);
      taken += __popc(eqm);
    }
  }
}

}  // namespace

// Every segment starts on a 16-byte boundary (the head states are float2,
// and max_seq may be odd).
inline size_t pad4(size_t n) { return (n + 3) / 4 * 4; }

size_t h2_workspace_floats(int B, int n_r, int G, int max_seq) {
  const size_t items = (size_t)B * n_r;
  // scores, importance, per-head (max, sum) states (float2), histograms (uint32)
  return pad4(items * (size_t)max_seq * G) + pad4(items * (size_t)max_seq) + pad4(items * G * 2) + items * kBins;
}

namespace {
struct H2Layout {
  float* scores;
  float* imp;
  float2* stats;
  uint32_t* hist;
};
H2Layout h2_layout(float* ws, int B, int n_r, int G, int max_seq) {
  const size_t items = (size_t)B * n_r;
  H2Layout l;
  l.scores = ws;
  l.imp = l.scores + pad4(items * (size_t)max_seq * G);
  l.stats = reinterpret_cast<float2*>(l.imp + pad4(items * (size_t)max_seq));
  l.hist = reinterpret_cast<uint32_t*>(reinterpret_cast<float*>(l.stats) + pad4(items * G * 2));
  return l;
}
}  // namespace

void h2_decode_outputs(float* ws, int B, int n_r, int G, int max_seq, float** scores, float2** stats) {
  const H2Layout l = h2_layout(ws, B, n_r, G, max_seq);
  *scores = l.scores;
  *stats = l.stats;
}

cudaError_t h2_workspace_clear(float* ws, int B, int n_r, int G, int max_seq, cudaStream_t s) {
  const H2Layout l = h2_layout(ws, B, n_r, G, max_seq);
  return cudaMemsetAsync(l.hist, 0, (size_t)B * n_r * kBins * sizeof(uint32_t), s);
}

cudaError_t launch_h2_topk(float* ws, int max_seq, const int32_t* lens, int B, int n_r, int G, int top_k,
                           int32_t* idx_out, cudaStream_t s) {
  if (B * n_r == 0) return cudaSuccess;
  if (G > 16) return cudaErrorInvalidValue;
  const H2Layout l = h2_layout(ws, B, n_r, G, max_seq);
  const size_t items = (size_t)B * n_r;
  const dim3 grid((max_seq + kChunk - 1) / kChunk, (unsigned)items);
  switch (G) {
#define AOH_IMP(g)                                                                                      \
  case g:                                                                                               \
    h2_imp_kernel<g><<<grid, kChunkThreads, 0, s>>>(l.scores, max_seq, lens, n_r, l.stats, l.imp, l.hist); \
    break;
    AOH_IMP(1) AOH_IMP(2) AOH_IMP(3) AOH_IMP(4) AOH_IMP(5) AOH_IMP(6) AOH_IMP(7) AOH_IMP(8) AOH_IMP(16)
#undef AOH_IMP
    default:
      return cudaErrorInvalidValue;
  }
  h2_select_kernel<<<(unsigned)items, kSelThreads, 0, s>>>(lens, n_r, max_seq, top_k, l.imp, l.hist, idx_out);
  return cudaGetLastError();
}

}  // namespace aoh
