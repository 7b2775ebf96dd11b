// Host-side declarations shared by the translation units of libaoh.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace aoh {

constexpr int kMaxKvHeads = 64;

// Bits of the device error word (and of the allocation-free entry point's
// sticky status word).
constexpr uint32_t kErrTimeout = 1u;   // a kernel's bounded wait ran out
constexpr uint32_t kErrCapacity = 2u;  // a decode step found a sequence already holding max_seq tokens

// Cache geometry as the kernels see it. Offsets are in bf16 elements from the
// cache base; see include/aoh.h for the layout.
struct CacheGeom {
  int B, Hq, Hkv, D, G;
  int max_seq, S, W;
  int K;  // streaming prefill eviction chunk; 0 = per-token window
  int n_r, n_s;
  // kind[h] = 0 retrieval / 1 streaming; idx[h] = index among heads of its kind
  uint8_t kind[kMaxKvHeads];
  uint8_t idx[kMaxKvHeads];
  uint8_t r_head[kMaxKvHeads];  // i-th retrieval head -> KV head
  uint8_t s_head[kMaxKvHeads];  // i-th streaming head -> KV head

  __host__ __device__ size_t r_region(int b, int i) const {
    return (size_t)(b * n_r + i) * 2 * (size_t)max_seq * D;
  }
  __host__ __device__ size_t s_region(int b, int i) const {
    return (size_t)B * n_r * 2 * (size_t)max_seq * D + (size_t)(b * n_s + i) * 2 * (size_t)(S + W) * D;
  }
  // K region start of (b, kv head); V follows after capacity rows.
  __host__ __device__ size_t region(int b, int h) const {
    return kind[h] ? s_region(b, idx[h]) : r_region(b, idx[h]);
  }
  __host__ __device__ int capacity(int h) const { return kind[h] ? S + W : max_seq; }
  // First non-sink key a streaming prefill row may see, for row i counted
  // from the start of the prefill call (calls start on chunk boundaries when
  // K > 0): the per-token window i - W + 1, or, with eviction after each
  // K-token chunk, the W positions before the row's chunk (Sec. 5,
  // "Chunked-Prefill Stage").
  __host__ __device__ int wstart(int i) const { return K ? (i / K) * K - W : i - W + 1; }
};

struct DecodeArgs {
  CUtensorMap tcr, tcs;  // cache regions (see PrefillTcArgs); read by the tcgen05 kernel
  CacheGeom geom;
  const void* q;      // [B][Hq][D]
  const void* k_new;  // [B][Hkv][D]
  const void* v_new;
  void* out;          // [B][Hq][D]
  void* kv;           // cache base
  int32_t* lens;      // [B] tokens held before this step (device)
  float* partials;    // [n_ctas][4][G][D + 2]: a CTA's own partial of its first / last
                      // shared item, then group partials of those items
  uint32_t* counters; // [B][n_r + n_s] group arrivals per item (items b-major, retrieval first)
  uint32_t* gcounters;  // [n_ctas][2] part arrivals per group (indexed by the group's first CTA)
  uint32_t* done;     // CTAs finished in this launch
  uint32_t* err;      // error word
  int n_ctas;         // CTAs sharing the rows of all items equally
  // nonzero: the launch's last CTA also leaves the error word and every
  // counter at zero after a timed-out launch, so the next launch needs no
  // clearing (the allocation-free entry point, which reports no timeouts)
  int self_clean = 0;
  // sticky status (or null): the last CTA ORs in the launch's kErrTimeout /
  // kErrCapacity flags; only the host clears it (allocation-free entry point)
  uint32_t* status = nullptr;
  // self-test (aoh_decode_step_noalloc_selftest; tcgen05 kernel), -1
  // otherwise: this CTA's softmax warps withhold their first P, so the MMA
  // warp's bounded wait for it runs out; every copy still lands, and the
  // launch's other CTAs finish as usual
  int stall_cta = -1;
  float scale_log2;   // log2(e) / sqrt(D)
  // H2Share anchor step (tcgen05 kernel): when non-null, every retrieval row's
  // scores (log2 units) go to scores[((b * n_r + i) * G + h) * score_stride + row],
  // and each retrieval head's final softmax state (max, sum of 2^(s - max))
  // to score_stats[(b * n_r + i) * G + h].
  float* scores = nullptr;
  int score_stride = 0;
  float2* score_stats = nullptr;
  // H2Share reuse step (both decode kernels): when non-null, retrieval item
  // (b, i) attends only to the cache rows idx[(b * n_idx_groups + idx_map[i]) *
  // top_k + r], r < min(top_k, t + 1).
  const int32_t* idx = nullptr;
  int top_k = 0;
  int n_idx_groups = 0;
  // Work units per row when the CTAs split the reuse step: gather_w for a
  // borrowed (gathered) row, ring_w for a contiguous one, so that a gathered
  // row weighs gather_w / ring_w contiguous rows; both 1 in other steps.
  int gather_w = 1;
  int ring_w = 1;
  // Work units charged ahead of each non-empty item's first row (the cost of
  // a CTA's switch to it), so the CTA that switches owns fewer rows.
  int item_cost = 0;
  uint8_t idx_map[kMaxKvHeads] = {};
};

struct AppendArgs {
  CacheGeom geom;
  const void* k;  // [B][T][Hkv][D]
  const void* v;
  void* kv;
  const int32_t* lens;  // device [B]: rows of the chunk
  const int32_t* base;  // device [B]: tokens cached before the chunk
  int T;
};

// Arguments of the tcgen05 prefill kernel: tensor maps over q / k / v
// ([B][T][H][D], box 128 rows x 64 columns, 128-byte swizzle) and a work list
// of (b, query head, first row) tiles sorted by cost.
struct PrefillTcArgs {
  CUtensorMap tq, tk, tv;  // the chunk's q / k / v
  CUtensorMap tcr, tcs;    // cache: retrieval / streaming regions as [regions][K, V][rows][D]
  CacheGeom geom;
  void* out;            // [B][T][Hq][D]
  const int32_t* lens;  // device [B]: rows of the chunk
  const int32_t* base;  // device [B]: tokens cached before the chunk
  const int4* work;     // {b, h, q0, cost}
  uint32_t* err;
  int T;
  float scale_log2;
};

// One warp waits on an mbarrier nothing arrives at, for limit_ns; the timeout
// lands in *err; *elapsed_ns receives how long the wait lasted (0 if it did
// not give up).
cudaError_t launch_wait_selftest(uint32_t* err, uint64_t limit_ns, unsigned long long* elapsed_ns, cudaStream_t s);

// cuTensorMapEncodeTiled from the driver (nullptr if unavailable).
PFN_cuTensorMapEncodeTiled_v12000 encode_fn();

// Store `msg` as the calling thread's aoh_last_error() message.
void record_error(const char* msg);

// Launchers (return the launch's cudaError_t).
bool prefill_tc_make_maps(PrefillTcArgs* a, const void* q, const void* k, const void* v, int B, int T);
bool prefill_tc_make_cache_maps(PrefillTcArgs* a, const void* kv);
// 4D maps over the retrieval / streaming regions of the cache at `kv`, as
// [regions][K, V][capacity rows][D] with box [1][1][128][64] and 128-byte
// swizzle; a kind with no heads leaves its map untouched.
bool make_cache_region_maps(CUtensorMap* tcr, CUtensorMap* tcs, const CacheGeom& g, const void* kv);
cudaError_t launch_prefill_tc(const PrefillTcArgs& a, int n_items, cudaStream_t s);
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t s);
// The CUDA-core decode kernel for any supported (D, G) (the H2Share reuse
// step takes this path at d_head 128 too), with its CTA count.
cudaError_t launch_decode_cc(const DecodeArgs& a, cudaStream_t s);
int decode_cc_ctas(long long total_rows, int num_sms);
bool decode_cc_supported(int D, int G);
// H2Share anchor selection after a decode step that wrote its scores to
// the start of `ws` ([B][n_r][G][stride] floats): per (sequence, retrieval
// head) the top_k positions by group importance. `ws` holds
// h2_workspace_floats() floats.
size_t h2_workspace_floats(int B, int n_r, int G, int max_seq);
// Where the decode kernel writes the scores (row stride `stride`, max_seq
// rounded up to a multiple of 4) and the per-head states in `ws`.
void h2_decode_outputs(float* ws, int B, int n_r, int G, int max_seq, float** scores, int* stride, float2** stats);
// One cluster launch computes the importances and selects; `lens` holds the
// lengths after the anchor step's append.
cudaError_t launch_h2_topk(float* ws, int max_seq, const int32_t* lens, int B, int n_r, int G, int top_k,
                           int32_t* idx_out, cudaStream_t s);
// CTAs for a decode launch over `total_rows` cached rows on `num_sms` SMs
// (the kernel is chosen by D and G).
int decode_ctas(long long total_rows, int num_sms, int D, int G);
// The tcgen05 decode kernel serves (D, G) (else the CUDA-core kernel does).
bool decode_uses_tc(int D, int G);
// Work units of a gathered row and of a contiguous row in the reuse step's
// split on the tcgen05 kernel (a borrowed K and V row copied by the gather
// warps against a contiguous row's share of a TMA tile stream), for group
// size G. Measured at 128K context, top_k 2048, half the KV heads streaming:
// gathered : contiguous = 3:2 / 5:3 / 2:1 / 3:1 gave 49 / 53 / 57 / - us at
// g = 4, B = 16 (4:3 55 us), and 33.5 / - / 35 / 37 us at g = 7, B = 16.
void reuse_tc_weights(int G, int* gather_w, int* ring_w);
// DecodeArgs::item_cost for a plain or anchor step of the tcgen05 kernel
// over total_rows rows on n_ctas CTAs of a num_sms-SM GPU (0 when each
// CTA's share is long).
int decode_tc_item_cost(long long total_rows, int n_ctas, int num_sms);
int decode_tc_ctas(long long total_rows, int num_sms);
cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t s);
// Floats of the partial buffer for `n_ctas` CTAs.
size_t decode_partial_floats(int n_ctas, int G, int D);
cudaError_t launch_append(const AppendArgs& a, cudaStream_t s);
cudaError_t launch_lens_add(int32_t* lens, const int32_t* add, int B, cudaStream_t s);
bool decode_supported(int D, int G);

}  // namespace aoh
