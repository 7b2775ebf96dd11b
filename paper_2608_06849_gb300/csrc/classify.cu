// Effective-rank head classifier (Sec. 4: Eq. 2-6 and Algorithm 1; Appendix
// "GQA Extension"), in fp64 on CUDA cores. It runs once per model, offline;
// exactness matters more than speed.
//
// For query head h with projections W_Q^h, W_K^h ([d_head][d_model]) the
// kernel attention matrix M_h = W_K^T W_Q (Eq. 2) has rank <= d_head, and
// its singular values are those of the d_head x d_head matrix
//   A = L_K^T L_Q,  with  W_Q W_Q^T = L_Q L_Q^T,  W_K W_K^T = L_K L_K^T
// (Cholesky factors; W^T = Q L^T is a thin QR, so M_h = Q_K (L_K^T L_Q) Q_Q^T).
// Steps:
//   1. gram_kernel: Gram matrices W W^T of every query and key projection
//      (bf16 products are exact in fp64; the d_model range is split over
//      CTAs and the parts are summed in a fixed order, so the result does
//      not depend on scheduling).
//   2. chol_kernel: semi-definite Cholesky in shared memory; a pivot at or
//      below d_head * eps * max(diag) leaves a zero column (rank deficiency).
//   3. er_kernel: A = L_K^T L_Q, then one-sided (Hestenes) Jacobi: pairs of
//      columns are rotated until every pair is orthogonal to d_head * eps,
//      with the round-robin ordering so the d_head / 2 pairs of a round
//      are disjoint; the singular values are the column norms. Values at or
//      below sigma_max * d_model * eps are the zeros of a rank-deficient
//      M_h and are dropped (Eq. 4 sums over nonzero values); ER (Eq. 4) is
//      exp of the entropy of the normalised singular values. FP64 is slow
//      on this part, so a pair costs one fp64 dot product and the column
//      update: squared norms are carried in shared memory (exact again at
//      each sweep), and the angle is formed in fp32 (any angle is exact).
//   4. classify_kernel: per layer, group score = mean ER of the group's
//      query heads; the k = ceil((100 - s) * groups / 100) lowest groups
//      (stable order, ties to the lower index) are retrieval, the rest
//      streaming.
// One call takes all layers of a model, so every matrix is a CTA of its own
// and the GPU fills up.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "../../include/aoh.h"
#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

using bf16 = __nv_bfloat16;
constexpr int kGT = 64;              // Gram output tile
constexpr int kGK = 32;              // d_model columns per step
constexpr int kGramThreads = 256;
constexpr int kMatThreads = 256;
constexpr int kMaxSweeps = 40;

// Matrices are numbered layer-major: layer l's query projections, then its
// key projections (nmat = Hq + Hkv per layer).
__device__ __forceinline__ const bf16* weight_of(const bf16* wq, const bf16* wk, int m, int Hq, int Hkv, int dh,
                                                 int dm) {
  const int nmat = Hq + Hkv, l = m / nmat, mi = m % nmat;
  return mi < Hq ? wq + ((size_t)l * Hq + mi) * dh * dm : wk + ((size_t)l * Hkv + (mi - Hq)) * dh * dm;
}

__global__ void __launch_bounds__(kGramThreads) gram_kernel(const bf16* wq, const bf16* wk, int Hq, int Hkv, int nall,
                                                            int dh, int dm, int span, double* part) {
  __shared__ double sa[kGK][kGT + 1], sb[kGK][kGT + 1];
  const int m = blockIdx.z, split = blockIdx.y;
  const int tiles = dh / kGT;
  const int ti = blockIdx.x / tiles, tj = blockIdx.x % tiles;
  const bf16* W = weight_of(wq, wk, m, Hq, Hkv, dh, dm);
  const int k0 = split * span, k1 = min(dm, k0 + span);
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  double acc[4][4] = {};
  for (int kc = k0; kc < k1; kc += kGK) {
    for (int e = threadIdx.x; e < kGT * kGK; e += kGramThreads) {
      const int row = e / kGK, kk = e % kGK;
      const bool in = kc + kk < k1;
      sa[kk][row] = in ? (double)__bfloat162float(W[(size_t)(ti * kGT + row) * dm + kc + kk]) : 0.0;
      sb[kk][row] = in ? (double)__bfloat162float(W[(size_t)(tj * kGT + row) * dm + kc + kk]) : 0.0;
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < kGK; ++kk) {
      double a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = sa[kk][ty * 4 + i];
        b[i] = sb[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fma(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  double* out = part + ((size_t)split * nall + m) * dh * dh;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) out[(size_t)(ti * kGT + ty * 4 + i) * dh + tj * kGT + tx * 4 + j] = acc[i][j];
}

// Sum of a block's values (every thread gets it); `red` holds 32 doubles.
__device__ double block_sum(double v, double* red) {
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  double s = 0.0;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
  return s;
}

__device__ double block_max(double v, double* red) {
  for (int o = 16; o >= 1; o >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  double s = red[0];
  for (int w = 1; w < (int)(blockDim.x >> 5); ++w) s = fmax(s, red[w]);
  return s;
}

// One matrix per CTA: G = sum of the split parts, then G = L L^T in place
// (lower triangle), written to L with the upper triangle zeroed.
__global__ void __launch_bounds__(kMatThreads) chol_kernel(const double* part, int nsplit, int nall, int dh,
                                                           double* L) {
  extern __shared__ double A[];  // [dh][dh] row-major
  __shared__ double red[32];
  __shared__ double inv_d;
  const int m = blockIdx.x;
  const size_t n2 = (size_t)dh * dh;
  for (int e = threadIdx.x; e < dh * dh; e += kMatThreads) {
    double s = 0.0;
    for (int p = 0; p < nsplit; ++p) s += part[((size_t)p * nall + m) * n2 + e];
    A[e] = s;
  }
  __syncthreads();
  double dmax = 0.0;
  for (int i = threadIdx.x; i < dh; i += kMatThreads) dmax = fmax(dmax, A[i * dh + i]);
  const double tol = dh * DBL_EPSILON * block_max(dmax, red);
  for (int j = 0; j < dh; ++j) {
    if (threadIdx.x == 0) {
      const double piv = A[j * dh + j];
      const double d = piv > tol ? sqrt(piv) : 0.0;
      A[j * dh + j] = d;
      inv_d = d > 0.0 ? 1.0 / d : 0.0;
    }
    __syncthreads();
    for (int i = j + 1 + threadIdx.x; i < dh; i += kMatThreads) A[i * dh + j] *= inv_d;
    __syncthreads();
    const int rem = dh - j - 1;
    for (int e = threadIdx.x; e < rem * rem; e += kMatThreads) {
      const int i = j + 1 + e / rem, k = j + 1 + e % rem;
      if (k <= i) A[i * dh + k] -= A[i * dh + j] * A[k * dh + j];
    }
    __syncthreads();
  }
  double* out = L + (size_t)m * n2;
  for (int e = threadIdx.x; e < dh * dh; e += kMatThreads) {
    const int i = e / dh, k = e % dh;
    out[e] = k <= i ? A[e] : 0.0;
  }
}

// Round-robin tournament: pair k of round r among n (even) columns.
__device__ __forceinline__ void rr_pair(int n, int r, int k, int& p, int& q) {
  if (k == 0) {
    p = n - 1;
    q = r;
  } else {
    p = (r + k) % (n - 1);
    q = (r - k + n - 1) % (n - 1);
  }
}

// Warp sum of a double (every lane gets it).
__device__ __forceinline__ double warp_sum(double v) {
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One query head per CTA (blockIdx.x = layer * Hq + head): A = L_K^T L_Q,
// one-sided Jacobi, ER.
__global__ void __launch_bounds__(kMatThreads) er_kernel(const double* L, int Hq, int Hkv, int dh, int dm,
                                                         double* er, int* sweeps_out) {
  extern __shared__ double A[];  // column-major: column c at A + c * dh; then dh squared norms
  __shared__ double red[32];
  __shared__ int rotated;
  const int hg = blockIdx.x, l = hg / Hq, h = hg % Hq, kv = h / (Hq / Hkv);
  const size_t n2 = (size_t)dh * dh;
  const double* Lq = L + ((size_t)l * (Hq + Hkv) + h) * n2;
  const double* Lk = L + ((size_t)l * (Hq + Hkv) + Hq + kv) * n2;
  double* nrm2 = A + n2;
  for (int e = threadIdx.x; e < dh * dh; e += kMatThreads) {
    const int i = e % dh, j = e / dh;  // A[i][j] = sum_m Lk[m][i] Lq[m][j] over m >= max(i, j)
    double s = 0.0;
    for (int mm = max(i, j); mm < dh; ++mm) s = fma(Lk[(size_t)mm * dh + i], Lq[(size_t)mm * dh + j], s);
    A[(size_t)j * dh + i] = s;
  }
  __syncthreads();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int kWarps = kMatThreads / 32;
  // a pair counts as orthogonal once |a_p . a_q| <= d_head * eps * |a_p| |a_q|
  // (the rounding level of a length-d_head dot product), tested squared
  const double rot_tol2 = (dh * DBL_EPSILON) * (dh * DBL_EPSILON);
  int sweep = 0;
  for (; sweep < kMaxSweeps; ++sweep) {
    // squared column norms, exact at the start of each sweep and carried
    // through its rotations
    for (int c = threadIdx.x; c < dh; c += kMatThreads) {
      const double* a = A + (size_t)c * dh;
      double s2 = 0.0;
      for (int i = 0; i < dh; ++i) s2 = fma(a[i], a[i], s2);
      nrm2[c] = s2;
    }
    if (threadIdx.x == 0) rotated = 0;
    __syncthreads();
    for (int r = 0; r < dh - 1; ++r) {
      for (int k = warp; k < dh / 2; k += kWarps) {
        int p, q;
        rr_pair(dh, r, k, p, q);
        double* ap = A + (size_t)p * dh;
        double* aq = A + (size_t)q * dh;
        const double al = nrm2[p], be = nrm2[q];
        double ga = 0.0;
        for (int i = lane; i < dh; i += 32) ga = fma(ap[i], aq[i], ga);
        ga = warp_sum(ga);
        if (ga != 0.0 && ga * ga > rot_tol2 * al * be) {
          // The angle only steers convergence: any (c, s) with c^2 + s^2 = 1
          // to fp64 precision is an exact orthogonal transform, so tan is
          // formed in fp32 and c, s from it in fp64.
          const float zeta = (float)(be - al) / (2.0f * (float)ga);
          const float tf = fabsf(zeta) > 1e18f ? 0.5f / zeta
                                               : copysignf(1.0f, zeta) / (fabsf(zeta) + sqrtf(1.0f + zeta * zeta));
          const double t = tf;
          const double c = rsqrt(1.0 + t * t), s = c * t;
          for (int i = lane; i < dh; i += 32) {
            const double x = ap[i], y = aq[i];
            ap[i] = fma(c, x, -s * y);
            aq[i] = fma(s, x, c * y);
          }
          if (lane == 0) {
            const double cc = c * c, ss = s * s, cs2 = 2.0 * c * s * ga;
            nrm2[p] = fmax(fma(cc, al, fma(ss, be, -cs2)), 0.0);
            nrm2[q] = fmax(fma(ss, al, fma(cc, be, cs2)), 0.0);
            rotated = 1;
          }
        }
      }
      __syncthreads();
    }
    const int any = rotated;
    __syncthreads();
    if (!any) break;
  }

  // singular values = column norms; ER over the nonzero ones (Eq. 4)
  double nrm = 0.0;
  if (threadIdx.x < dh) {
    const double* a = A + (size_t)threadIdx.x * dh;
    for (int i = 0; i < dh; ++i) nrm = fma(a[i], a[i], nrm);
    nrm = sqrt(nrm);
  }
  const double smax = block_max(threadIdx.x < dh ? nrm : 0.0, red);
  const double tol = smax * (double)max(dm, dh) * DBL_EPSILON;
  const bool keep = threadIdx.x < dh && nrm > tol;
  const double total = block_sum(keep ? nrm : 0.0, red);
  double ent = 0.0;
  if (keep) {
    const double p = nrm / total;
    ent = -p * log(p);
  }
  ent = block_sum(ent, red);
  if (threadIdx.x == 0) {
    er[hg] = exp(ent);
    sweeps_out[hg] = sweep;
  }
}

// One layer per block (blockIdx.x), one thread.
__global__ void classify_kernel(const double* er_all, int Hq, int Hkv, int sparsity_pct, uint8_t* labels_all) {
  if (threadIdx.x != 0) return;
  const double* er = er_all + (size_t)blockIdx.x * Hq;
  uint8_t* labels = labels_all + (size_t)blockIdx.x * Hkv;
  const int g = Hq / Hkv;
  double score[kMaxKvHeads];
  int order[kMaxKvHeads];
  for (int kv = 0; kv < Hkv; ++kv) {
    double s = 0.0;
    for (int i = 0; i < g; ++i) s += er[kv * g + i];
    score[kv] = s / g;
    order[kv] = kv;
  }
  for (int i = 1; i < Hkv; ++i) {  // stable insertion sort, ascending
    const int x = order[i];
    int j = i - 1;
    while (j >= 0 && score[order[j]] > score[x]) {
      order[j + 1] = order[j];
      --j;
    }
    order[j + 1] = x;
  }
  const int k = ((100 - sparsity_pct) * Hkv + 99) / 100;
  for (int i = 0; i < Hkv; ++i) labels[order[i]] = i < k ? AOH_RETRIEVAL : AOH_STREAMING;
}

}  // namespace
}  // namespace aoh

using namespace aoh;

extern "C" aoh_status aoh_classify(const void* w_q, const void* w_k, int32_t n_layers, int32_t n_q_heads,
                                   int32_t n_kv_heads, int32_t d_head, int32_t d_model, int32_t sparsity_pct,
                                   double* er_out, uint8_t* labels_out, void* stream) {
  auto fail = [](aoh_status st, const char* msg) {
    record_error(msg);
    return st;
  };
  if (!w_q || !w_k || !labels_out)
    return fail(AOH_ERR_INVALID, "aoh_classify: w_q, w_k and labels_out must not be NULL");
  if (n_layers < 1 || n_layers > 65535) return fail(AOH_ERR_INVALID, "aoh_classify: n_layers outside [1, 65535]");
  if (n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads)
    return fail(AOH_ERR_INVALID, "aoh_classify: n_q_heads must be a positive multiple of n_kv_heads");
  if (n_kv_heads > kMaxKvHeads) return fail(AOH_ERR_UNSUPPORTED, "aoh_classify: more than 64 KV heads");
  if (d_head != 64 && d_head != 128) return fail(AOH_ERR_UNSUPPORTED, "aoh_classify: d_head must be 64 or 128");
  if (d_model < 1) return fail(AOH_ERR_INVALID, "aoh_classify: d_model must be >= 1");
  if (sparsity_pct < 0 || sparsity_pct > 100)
    return fail(AOH_ERR_INVALID, "aoh_classify: sparsity_pct outside [0, 100]");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int dh = d_head, nmat = n_q_heads + n_kv_heads, tiles = dh / kGT;
  const int nall = n_layers * nmat, nq = n_layers * n_q_heads;
  if ((long long)n_layers * nmat > 65535) return fail(AOH_ERR_INVALID, "aoh_classify: too many matrices in one call");
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return fail(AOH_ERR_CUDA, "aoh_classify: device query failed");
  // split d_model so that the Gram grid covers about two waves, >= 256 columns a split
  int nsplit = (2 * sms + nall * tiles * tiles - 1) / (nall * tiles * tiles);
  nsplit = std::max(1, std::min(nsplit, std::max(1, d_model / 256)));
  nsplit = std::min(nsplit, 16);
  const int span = ((d_model + nsplit - 1) / nsplit + kGK - 1) / kGK * kGK;
  nsplit = (d_model + span - 1) / span;
  const size_t n2 = (size_t)dh * dh;
  const size_t bytes = ((size_t)nsplit * nall * n2 + (size_t)nall * n2 + nq) * sizeof(double) + nq * sizeof(int) +
                       (size_t)n_layers * n_kv_heads + 64;
  void* scratch = nullptr;
  e = cudaMallocAsync(&scratch, bytes, s);
  if (e != cudaSuccess) return fail(AOH_ERR_CUDA, "aoh_classify: cudaMallocAsync failed");
  double* part = static_cast<double*>(scratch);
  double* L = part + (size_t)nsplit * nall * n2;
  double* er = L + (size_t)nall * n2;
  int* sweeps = reinterpret_cast<int*>(er + nq);
  uint8_t* labels = reinterpret_cast<uint8_t*>(sweeps + nq);
  const int smem = (int)(n2 * sizeof(double));
  const int smem_er = (int)((n2 + dh) * sizeof(double));
  static bool attr_set = false;
  if (!attr_set) {
    e = cudaFuncSetAttribute(chol_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 128 * 128 * 8);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(er_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (128 * 128 + 128) * 8);
    if (e != cudaSuccess) {
      cudaFreeAsync(scratch, s);
      return fail(AOH_ERR_CUDA, "aoh_classify: cudaFuncSetAttribute failed");
    }
    attr_set = true;
  }
  gram_kernel<<<dim3(tiles * tiles, nsplit, nall), kGramThreads, 0, s>>>(static_cast<const bf16*>(w_q),
                                                                          static_cast<const bf16*>(w_k), n_q_heads,
                                                                          n_kv_heads, nall, dh, d_model, span, part);
  chol_kernel<<<nall, kMatThreads, smem, s>>>(part, nsplit, nall, dh, L);
  er_kernel<<<nq, kMatThreads, smem_er, s>>>(L, n_q_heads, n_kv_heads, dh, d_model, er, sweeps);
  classify_kernel<<<n_layers, 32, 0, s>>>(er, n_q_heads, n_kv_heads, sparsity_pct, labels);
  e = cudaGetLastError();
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(labels_out, labels, (size_t)n_layers * n_kv_heads, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess && er_out) e = cudaMemcpyAsync(er_out, er, nq * sizeof(double), cudaMemcpyDeviceToHost, s);
  const cudaError_t f = cudaFreeAsync(scratch, s);
  if (e == cudaSuccess) e = f;
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(AOH_ERR_CUDA, "aoh_classify: a CUDA call failed");
  return AOH_OK;
}
