// H2Share head mapping (the paper's H2Share section, Eq. sim, and its GQA
// extension appendix), offline, from frozen weights. For anchor query head
// h (KV group g) and reuse query head h' (KV group g'):
//   sim(h, h') = tr(A B) / sqrt(n_a(h) n_r(h')),
//   A = W_Qa^h W_Qr^h'^T,  B = W_Kr^g' W_Ka^g^T            (d_head x d_head),
//   n_a(h) = tr((W_Qa^h W_Qa^h^T)(W_Ka^g W_Ka^g^T)), n_r likewise,
// the normalised Frobenius inner product of the two kernel matrices
// M = W_K^T W_Q through the trace identities. Group similarity is the mean
// over the two groups' query-head pairs; every reuse retrieval group maps to
// the anchor retrieval group of highest similarity (ties to the lower index).
//
// All d_head x d_head products come from dense bf16 contractions C = A B^T
// over d_model on tcgen05, in two launches of gemm_kernel:
//   1. the key side, stored (small: [Hkv d_head]^2 each):
//        Y = K_r K_a^T,  G_ka = K_a K_a^T,  G_kr = K_r K_r^T;
//   2. the query side, never stored: X = Q_a Q_r^T (every A above) and the
//      diagonal tiles of Q_a Q_a^T and Q_r Q_r^T leave TMEM straight into the
//      trace. Row i of a tile sits in TMEM lane i, so the thread holding it
//      multiplies its 32-column chunk by the matching key-side block read
//      transposed (Y[g' d_head + j][g d_head + i]: consecutive i across the
//      warp, coalesced), and one fp64 partial per 32 x 32 block is written.
// map_kernel then sums the partials of each head pair in a fixed order (the
// result does not depend on scheduling), forms the group means and takes the
// argmax.
//
// gemm_kernel: one CTA per 128 x 128 output tile, several problems per
// launch (blockIdx ranges), 192 threads: warp 0 TMA (2D tensor maps, 128-byte
// swizzle, 64 columns of d_model per step, 3-stage ring; rows and columns
// past the matrix read as zeros), warp 1 TMEM owner and MMA issuer
// (kind::f16, both operands K-major, fp32 accumulator in TMEM), warps 2-5 the
// epilogue. 97 KB of shared memory and 128 TMEM columns let two CTAs share an
// SM, so one CTA's epilogue overlaps the other's main loop.
#include <math.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/aoh.h"
#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace aoh {
namespace {

constexpr int kTM = 128;             // output tile
constexpr int kTK = 64;              // d_model columns per step
constexpr int kStages = 3;
constexpr int kGemmThreads = 192;
constexpr int kTileBytes = kTM * kTK * 2;  // 16 KB
constexpr int GEMM_SMEM = kStages * 2 * kTileBytes + 256 + 1024;
constexpr int kMaxProblems = 3;
constexpr uint32_t IDESC = idesc_bf16(kTM, kTM, false);

struct Problem {
  CUtensorMap ta, tb;  // A [M][K], B [N][K], bf16, row-major
  float* c;            // store mode: C [M][N] fp32
  const float* r;      // trace mode: key-side matrix, leading dimension ldr
  double* out;         // trace mode: per head pair tr(A B), out[h * (N / d_head) + h']
  int out_diag;        // trace mode: only pairs h == h', to out[h]
  int M, N, ldr;
  int diag;            // only tiles (t, t)
  int tiles;           // CTAs of this problem
};

struct GemmArgs {
  Problem p[kMaxProblems];
  int n_problems, K;
  int trace;           // 0: store C; 1: block traces against r
  int dh, group;       // d_head; query heads per KV group
  uint32_t* err;
};

__global__ void __launch_bounds__(kGemmThreads, 2) gemm_kernel(const __grid_constant__ GemmArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kTileBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + 2 * kStages * kTileBytes);
  uint64_t* empty = full + kStages;
  uint64_t* done = empty + kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int pid = 0, t = blockIdx.x;
  while (pid + 1 < a.n_problems && t >= a.p[pid].tiles) {
    t -= a.p[pid].tiles;
    ++pid;
  }
  const Problem& P = a.p[pid];
  const int tiles_n = (P.N + kTM - 1) / kTM;
  const int tm = P.diag ? t : t / tiles_n;
  const int tn = P.diag ? t : t % tiles_n;
  const int nk = (a.K + kTK - 1) / kTK;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 128);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  __shared__ double red[4][4];  // trace mode: [row quarter][column chunk] partials of the tile
  // the next launch on the stream (the query side after the key side) may
  // start its main loop now; it waits for this grid only before its epilogue
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&P.ta);
      prefetch_tmap(&P.tb);
      int issued = 0;
      for (int kc = 0; kc < nk; ++kc) {
        const int st = kc % kStages;
        if (kc >= kStages && !wait_bar(&empty[st], ((kc / kStages) & 1) ^ 1, a.err, abort_flag)) break;
        mbar_arrive_expect_tx(&full[st], 2 * kTileBytes);
        tma_load_2d(sA + st * kTileBytes, &P.ta, kc * kTK, tm * kTM, &full[st]);
        tma_load_2d(sB + st * kTileBytes, &P.tb, kc * kTK, tn * kTM, &full[st]);
        issued = kc + 1;
      }
      // no copy may still be in flight when the CTA exits
      for (int j = issued > kStages ? issued - kStages : 0; j < issued; ++j)
        drain_wait(&full[j % kStages], (j / kStages) & 1, a.err);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      for (int kc = 0; kc < nk; ++kc) {
        const int st = kc % kStages;
        if (!wait_bar(&full[st], (kc / kStages) & 1, a.err, abort_flag)) break;
        tc_fence_after();
        const uint32_t aa = smem_u32(sA + st * kTileBytes), bb = smem_u32(sB + st * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kTK / 16; ++kk)
          tc_mma(tmem, sdesc_sw128(aa + kk * 32, 16, 1024), sdesc_sw128(bb + kk * 32, 16, 1024), IDESC,
                 (kc > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&empty[st]);
      }
      tc_commit(done);
      drain_wait(done, 0, a.err);  // this warp frees TMEM: its MMAs must be done
    }
  } else {
    // epilogue: warp w reads TMEM lanes 32 * (w % 4) .. + 31, rows of the
    // tile. M and N are multiples of 32, so a warp's rows and a 32-column
    // chunk are either all inside the matrix or all past it.
    const int q4 = warp & 3;
    const bool ok = __all_sync(0xffffffffu, wait_bar(done, 0, a.err, abort_flag));
    const int row0 = tm * kTM + q4 * 32;
    // trace mode reads the key-side matrices of the previous launch
    if (a.trace) {
      asm volatile("griddepcontrol.wait;" ::: "memory");
      if (lane < 4) red[q4][lane] = 0.0;
      __syncwarp();
    }
    if (ok && row0 < P.M) {
      tc_fence_after();
      const int r = row0 + lane;
      const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
      const int h = r / a.dh, i = r % a.dh, g = h / a.group;
#pragma unroll 1
      for (int c = 0; c < kTM / 32; ++c) {
        const int col0 = tn * kTM + c * 32;
        if (col0 >= P.N) break;
        uint32_t v[32];
        tmem_ld32(tl + c * 32, v);
        tmem_ld_wait();
        if (a.trace) {
          // sum_j X[i][j] * R[g' d_head + j][g d_head + i] over this chunk's
          // 32 columns j (all of one head h'), fp32 products in four
          // interleaved partial sums, then fp64
          const int hp = col0 / a.dh, j0 = col0 % a.dh, gp = hp / a.group;
          const float* rp = P.r + (size_t)(gp * a.dh + j0) * P.ldr + g * a.dh + i;
          float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int e = 0; e < 32; ++e) s[e & 3] = fmaf(__uint_as_float(v[e]), rp[(size_t)e * P.ldr], s[e & 3]);
          double acc = ((double)s[0] + (double)s[1]) + ((double)s[2] + (double)s[3]);
#pragma unroll
          for (int o = 16; o >= 1; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
          if (lane == 0) red[q4][c] = acc;
        } else {
          float* dst = P.c + (size_t)r * P.N + col0;
#pragma unroll
          for (int e = 0; e < 32; e += 4)
            *reinterpret_cast<float4*>(dst + e) = make_float4(__uint_as_float(v[e]), __uint_as_float(v[e + 1]),
                                                              __uint_as_float(v[e + 2]), __uint_as_float(v[e + 3]));
        }
      }
    }
    if (a.trace) {
      // the tile holds whole head pairs (128 / d_head heads a side); each
      // pair's trace is the sum of its 32 x 32 blocks, rows then columns
      named_barrier_sync(1, 128);
      if (threadIdx.x == 64) {
        const int R = kTM / a.dh, W = a.dh / 32, Hr = P.M / a.dh, Hc = P.N / a.dh;
        for (int ha = 0; ha < R; ++ha)
          for (int hb = 0; hb < R; ++hb) {
            const int h = tm * R + ha, hp = tn * R + hb;
            if (h >= Hr || hp >= Hc || (P.out_diag && h != hp)) continue;
            double sum = 0.0;
            for (int x = 0; x < W; ++x)
              for (int y = 0; y < W; ++y) sum += red[ha * W + x][hb * W + y];
            P.out[P.out_diag ? h : (size_t)h * Hc + hp] = sum;
          }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 128);
}

// 2D map over a row-major [rows][K] bf16 matrix, box 128 rows x 64 columns.
bool make_2d_map(CUtensorMap* map, const void* base, int rows, int K) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  cuuint32_t box[2] = {kTK, kTM};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One problem of a launch: C = A B^T with A [M][K], B [N][K].
bool add_problem(GemmArgs& g, const void* A, int M, const void* B, int N, int K, bool diag, float* c,
                 const float* r, int ldr, double* out) {
  Problem& p = g.p[g.n_problems++];
  if (!make_2d_map(&p.ta, A, M, K) || !make_2d_map(&p.tb, B, N, K)) return false;
  p.c = c;
  p.r = r;
  p.out = out;
  p.out_diag = diag ? 1 : 0;
  p.M = M;
  p.N = N;
  p.ldr = ldr;
  p.diag = diag ? 1 : 0;
  const int tiles_m = (M + kTM - 1) / kTM, tiles_n = (N + kTM - 1) / kTM;
  p.tiles = diag ? std::min(tiles_m, tiles_n) : tiles_m * tiles_n;
  return true;
}

// A trace-mode launch overlaps the key-side launch before it (programmatic
// dependent launch): only its epilogue waits for that grid.
cudaError_t launch_gemm(const GemmArgs& g, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, GEMM_SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  int grid = 0;
  for (int i = 0; i < g.n_problems; ++i) grid += g.p[i].tiles;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kGemmThreads);
  cfg.dynamicSmemBytes = GEMM_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g.trace ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_kernel, g);
}

struct Labels {
  uint8_t a[kMaxKvHeads], r[kMaxKvHeads];
};

// sim(h, h') = tr(A B) / sqrt(n_a(h) n_r(h')) from the traces, then the
// group means and the argmax. fp64 divides and square roots are slow on this
// part: 2 Hq of them (the inverse norms), spread over the block's threads.
__global__ void map_kernel(const double* num, const double* na, const double* nr, int Hq, int Hkv, Labels lab,
                           double* inv, double* sim, double* gsim, int32_t* map) {
  const int g = Hq / Hkv;
  for (int id = threadIdx.x; id < 2 * Hq; id += blockDim.x) inv[id] = 1.0 / sqrt(id < Hq ? na[id] : nr[id - Hq]);
  __syncthreads();
  for (int id = threadIdx.x; id < Hq * Hq; id += blockDim.x) sim[id] = num[id] * inv[id / Hq] * inv[Hq + id % Hq];
  __syncthreads();
  for (int id = threadIdx.x; id < Hkv * Hkv; id += blockDim.x) {
    const int ga = id / Hkv, gr = id % Hkv;
    double s = 0.0;
    for (int i = 0; i < g; ++i)
      for (int j = 0; j < g; ++j) s += sim[(ga * g + i) * Hq + gr * g + j];
    gsim[id] = s / (g * g);
  }
  __syncthreads();
  for (int gr = threadIdx.x; gr < Hkv; gr += blockDim.x) {
    int best = -1;
    if (lab.r[gr] == AOH_RETRIEVAL)
      for (int ga = 0; ga < Hkv; ++ga)
        if (lab.a[ga] == AOH_RETRIEVAL && (best < 0 || gsim[ga * Hkv + gr] > gsim[best * Hkv + gr])) best = ga;
    map[gr] = best;
  }
}

// One workspace per device, grown on demand and kept for the process (a
// stream-ordered allocation per call would be mapped and released at every
// synchronise); calls on one device are serialised by the mutex, and each
// synchronises its stream before returning, so the next may reuse it.
constexpr int kWsDevices = 64;
std::mutex g_ws_mutex;
void* g_ws[kWsDevices] = {};
size_t g_ws_cap[kWsDevices] = {};

}  // namespace
}  // namespace aoh

using namespace aoh;

extern "C" aoh_status aoh_h2share_map(const void* w_q_anchor, const void* w_k_anchor, const void* w_q_reuse,
                                      const void* w_k_reuse, int32_t n_q_heads, int32_t n_kv_heads, int32_t d_head,
                                      int32_t d_model, const uint8_t* anchor_labels, const uint8_t* reuse_labels,
                                      int32_t* map_out, double* group_sim_out, void* stream) {
  auto fail = [](aoh_status st, const char* msg) {
    record_error(msg);
    return st;
  };
  if (!w_q_anchor || !w_k_anchor || !w_q_reuse || !w_k_reuse || !anchor_labels || !reuse_labels || !map_out)
    return fail(AOH_ERR_INVALID, "aoh_h2share_map: NULL argument");
  if (n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads)
    return fail(AOH_ERR_INVALID, "aoh_h2share_map: n_q_heads must be a positive multiple of n_kv_heads");
  if (n_kv_heads > kMaxKvHeads) return fail(AOH_ERR_UNSUPPORTED, "aoh_h2share_map: more than 64 KV heads");
  if (d_head != 64 && d_head != 128) return fail(AOH_ERR_UNSUPPORTED, "aoh_h2share_map: d_head must be 64 or 128");
  if (d_model < 8 || d_model % 8) return fail(AOH_ERR_INVALID, "aoh_h2share_map: d_model must be a multiple of 8");
  const uintptr_t al = reinterpret_cast<uintptr_t>(w_q_anchor) | reinterpret_cast<uintptr_t>(w_k_anchor) |
                       reinterpret_cast<uintptr_t>(w_q_reuse) | reinterpret_cast<uintptr_t>(w_k_reuse);
  if (al % 16) return fail(AOH_ERR_INVALID, "aoh_h2share_map: weights must be 16-byte aligned");
  Labels lab;
  for (int i = 0; i < n_kv_heads; ++i) {
    if (anchor_labels[i] > 1 || reuse_labels[i] > 1) return fail(AOH_ERR_INVALID, "aoh_h2share_map: bad label");
    lab.a[i] = anchor_labels[i];
    lab.r[i] = reuse_labels[i];
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int Hq = n_q_heads, Hkv = n_kv_heads, dh = d_head, dm = d_model;
  const int nq = Hq * dh, nk = Hkv * dh;
  // key-side Y, G_ka, G_kr; traces (pairs, two norm sets); inverse norms;
  // head and group similarities; map; error word
  const size_t bytes = 3 * (size_t)nk * nk * 4 + ((size_t)Hq * Hq + 2 * Hq) * 8 + 2 * (size_t)Hq * 8 +
                       (size_t)Hq * Hq * 8 + (size_t)Hkv * Hkv * 8 + Hkv * 4 + 256;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kWsDevices) return fail(AOH_ERR_CUDA, "aoh_h2share_map: no usable device");
  std::lock_guard<std::mutex> lock(g_ws_mutex);
  if (g_ws_cap[dev] < bytes) {
    if (g_ws[dev]) cudaFree(g_ws[dev]);
    g_ws[dev] = nullptr;
    g_ws_cap[dev] = 0;
    e = cudaMalloc(&g_ws[dev], bytes);
    if (e != cudaSuccess) return fail(AOH_ERR_CUDA, "aoh_h2share_map: workspace allocation failed");
    g_ws_cap[dev] = bytes;
  }
  void* ws = g_ws[dev];
  float* Y = static_cast<float*>(ws);
  float* gka = Y + (size_t)nk * nk;
  float* gkr = gka + (size_t)nk * nk;
  double* num = reinterpret_cast<double*>(gkr + (size_t)nk * nk);
  double* na = num + (size_t)Hq * Hq;
  double* nr = na + Hq;
  double* inv = nr + Hq;
  double* sim = inv + 2 * (size_t)Hq;
  double* gsim = sim + (size_t)Hq * Hq;
  int32_t* map = reinterpret_cast<int32_t*>(gsim + (size_t)Hkv * Hkv);
  uint32_t* err = reinterpret_cast<uint32_t*>(map + Hkv);
  GemmArgs kg{}, qg{};
  kg.K = qg.K = dm;
  kg.dh = qg.dh = dh;
  kg.group = qg.group = Hq / Hkv;
  kg.err = qg.err = err;
  kg.trace = 0;
  qg.trace = 1;
  bool maps_ok = add_problem(kg, w_k_reuse, nk, w_k_anchor, nk, dm, false, Y, nullptr, 0, nullptr) &&
                 add_problem(kg, w_k_anchor, nk, w_k_anchor, nk, dm, false, gka, nullptr, 0, nullptr) &&
                 add_problem(kg, w_k_reuse, nk, w_k_reuse, nk, dm, false, gkr, nullptr, 0, nullptr) &&
                 add_problem(qg, w_q_anchor, nq, w_q_reuse, nq, dm, false, nullptr, Y, nk, num) &&
                 add_problem(qg, w_q_anchor, nq, w_q_anchor, nq, dm, true, nullptr, gka, nk, na) &&
                 add_problem(qg, w_q_reuse, nq, w_q_reuse, nq, dm, true, nullptr, gkr, nk, nr);
  if (!maps_ok) e = cudaErrorInvalidValue;
  if (e == cudaSuccess) e = cudaMemsetAsync(err, 0, 4, s);
  if (e == cudaSuccess) e = launch_gemm(kg, s);
  if (e == cudaSuccess) e = launch_gemm(qg, s);
  if (e == cudaSuccess) {
    map_kernel<<<1, 1024, 0, s>>>(num, na, nr, Hq, Hkv, lab, inv, sim, gsim, map);
    e = cudaGetLastError();
  }
  // group similarities, map and error word are contiguous: one copy back
  const size_t res_bytes = (size_t)Hkv * Hkv * 8 + (size_t)Hkv * 4 + 4;
  std::vector<unsigned char> res(res_bytes);
  if (e == cudaSuccess) e = cudaMemcpyAsync(res.data(), gsim, res_bytes, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(AOH_ERR_CUDA, "aoh_h2share_map: a CUDA call failed");
  uint32_t h_err = 0;
  memcpy(map_out, res.data() + (size_t)Hkv * Hkv * 8, (size_t)Hkv * 4);
  if (group_sim_out) memcpy(group_sim_out, res.data(), (size_t)Hkv * Hkv * 8);
  memcpy(&h_err, res.data() + (size_t)Hkv * Hkv * 8 + (size_t)Hkv * 4, 4);
  if (h_err) return fail(AOH_ERR_TIMEOUT, "aoh_h2share_map: a kernel's bounded wait ran out");
  return AOH_OK;
}
