// Pieces shared by the two decode kernels (CUDA cores, tcgen05): the
// stream-K split of a step's cached rows over the CTAs of a launch, and the
// merge of an item's split partials (Sec. 5 "Decode Stage": each head's
// softmax over its visible positions, assembled from per-split
// log-sum-exp states).
//
// An item is one (sequence b, KV head) pair; items are ordered b-major, the
// retrieval heads of a sequence before its streaming heads. The rows of all
// items are concatenated and CTA p of P takes rows [p*T/P, (p+1)*T/P).
#pragma once

#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace dec {

constexpr int kGroup = 16;  // parts merged per first-level group

// Tokens held by sequence b before this step: from the kernel's shared
// memory copy of the lengths when it has one (`lens_s`), else from global
// memory. Under a saturated HBM stream even an L2 hit costs microseconds,
// which at an item switch would stall the TMA ring.
__device__ __forceinline__ int seq_len(const DecodeArgs& a, int b, const int* lens_s) {
  return lens_s ? lens_s[b] : __ldcg(&a.lens[b]);
}

// A sequence whose retrieval heads are already full (t >= max_seq) cannot
// take the new token: the step skips every item of it (nothing appended,
// no output written) and the launch's last CTA leaves its length as it is
// and flags kErrCapacity. The host checks its mirror of the lengths before
// a handle launch; this guard covers callers whose host bound can go stale
// (the allocation-free entry point, e.g. replayed from a CUDA graph).
__device__ __forceinline__ bool seq_full(const CacheGeom& g, int t) { return g.n_r > 0 && t >= g.max_seq; }

// Rows of item `id`. Retrieval: t + 1 rows (min(top_k, t + 1) borrowed rows
// in the H2Share reuse step); streaming: min(t + 1, S + W) ring rows;
// t = tokens held before this step. 0 for every item of a full sequence.
__device__ __forceinline__ int item_rows(const DecodeArgs& a, int id, const int* lens_s = nullptr) {
  const CacheGeom& g = a.geom;
  const int HK = g.n_r + g.n_s;
  const int b = id / HK, k = id - b * HK;
  const int t = seq_len(a, b, lens_s);
  if (seq_full(g, t)) return 0;
  if (k < g.n_r) return a.idx ? min(a.top_k, t + 1) : t + 1;
  return min(t + 1, g.S + g.W);
}

// Work units of item `id`: its rows, weighted in the reuse step by gather_w
// (gathered rows) and ring_w (contiguous rows). The CTAs split the units
// equally.
__device__ __forceinline__ int item_weight(const DecodeArgs& a, int id) {
  if (a.idx == nullptr) return 1;
  return id % (a.geom.n_r + a.geom.n_s) < a.geom.n_r ? a.gather_w : a.ring_w;
}
// A non-empty item also carries a.item_cost units ahead of its first row:
// the cost of switching to it, charged to the CTA whose range holds its
// start.
__device__ __forceinline__ long long item_units(const DecodeArgs& a, int id, const int* lens_s = nullptr) {
  const int rows = item_rows(a, id, lens_s);
  return rows > 0 ? (long long)rows * item_weight(a, id) + a.item_cost : 0;
}

// The rows of item `id` (at unit offset off) that the CTA with unit range
// [start, end) owns: row r sits at unit off + cost + r * w, so every row
// belongs to exactly one CTA. lo >= hi when the CTA owns none.
struct Span {
  int rows, w, cost, lo, hi;
  long long units;
};
__device__ __forceinline__ Span item_span(const DecodeArgs& a, int id, const int* lens_s, long long off,
                                          long long start, long long end) {
  Span s;
  s.rows = item_rows(a, id, lens_s);
  s.w = item_weight(a, id);
  s.cost = s.rows > 0 ? a.item_cost : 0;
  s.units = (long long)s.rows * s.w + s.cost;
  const long long base = off + s.cost;
  const long long ulo = max(start, base) - base, uhi = min(end, base + (long long)s.rows * s.w) - base;
  s.lo = (int)((ulo + s.w - 1) / s.w);
  s.hi = uhi > ulo ? (int)((uhi + s.w - 1) / s.w) : s.lo;
  return s;
}

// CTA whose row range contains global row x.
__device__ __forceinline__ int cta_of(long long x, long long total, int P) {
  return (int)(((x + 1) * (long long)P - 1) / total);
}

// Block-wide prefix sum of the items' rows (warp shuffles, then the warp
// totals; up to 32 items, warp 0 alone, with no block barrier, which saves
// ~0.4 us of a short step). On return (after the caller's next
// __syncthreads) sh64[0] = total rows, sh64[1] = first row of the first item
// this CTA touches, sh32[0] = that item. `wsum` is THREADS / 32 longs of
// scratch shared memory.
template <int THREADS>
__device__ __forceinline__ void find_cta_range(const DecodeArgs& a, long long* wsum, long long* sh64, int* sh32,
                                               const int* lens_s = nullptr) {
  constexpr int NW = THREADS / 32;
  const CacheGeom& g = a.geom;
  const int n_items = g.B * (g.n_r + g.n_s);
  const int P = a.n_ctas, p = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (n_items <= 32) {
    // few items: warp 0 scans them alone (lane i holds item i)
    if (warp == 0) {
      const long long u = lane < n_items ? item_units(a, lane, lens_s) : 0;
      long long inc = u;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
      }
      const long long total = __shfl_sync(0xffffffffu, inc, 31);
      const long long start = (long long)p * total / P;
      const unsigned past = __ballot_sync(0xffffffffu, lane < n_items && inc > start);
      const int first = past ? __ffs(past) - 1 : n_items;
      const long long excl = __shfl_sync(0xffffffffu, inc - u, first < 32 ? first : 31);
      if (lane == 0) {
        sh64[0] = total;
        sh32[0] = first;
        sh64[1] = first < n_items ? excl : total;
      }
    }
    return;
  }
  const int per = (n_items + THREADS - 1) / THREADS;
  const int i0 = min(n_items, (int)threadIdx.x * per), i1 = min(n_items, i0 + per);
  long long mine = 0;
  for (int id = i0; id < i1; ++id) mine += item_units(a, id, lens_s);
  long long inc = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long run = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const long long v = wsum[w];
      wsum[w] = run;
      run += v;
    }
    sh64[0] = run;
    sh32[0] = n_items;
    sh64[1] = run;
  }
  __syncthreads();
  const long long total = sh64[0];
  const long long start = (long long)p * total / P;
  long long off = wsum[warp] + inc - mine;
  if (i0 < i1 && off <= start && start < off + mine) {
    int id = i0;
    while (true) {
      const long long r = item_units(a, id, lens_s);
      if (start < off + r) break;
      off += r;
      ++id;
    }
    sh32[0] = id;
    sh64[1] = off;
  }
}

// Partial state of split CTA q for an item whose first CTA is f: o[G][D]
// (unnormalised), then m[G] (running max, log2 units), then l[G], in slots
// of partial_stride floats (16-byte aligned). Slot 0/1: the CTA's first /
// last shared item; slot 2/3: the group partial of the group the CTA heads.
__host__ __device__ constexpr int partial_stride(int G, int D) { return (G * (D + 2) + 3) / 4 * 4; }

__device__ __forceinline__ float* partial_slot(const DecodeArgs& a, int q, int slot, int G, int D) {
  return a.partials + ((size_t)q * 4 + slot) * (size_t)partial_stride(G, D);
}

// Merge n partial states (part(j) returns the j-th) with log-sum-exp
// weights. Writes the normalised bf16 output to `out` (and, if `stats` is
// given, the merged (max, sum) of every head to stats[0..G)), or the merged
// partial to `dst`. Run by NT threads that share named barrier 1. The partials sit
// in L2, so the merge is a chain of L2 round trips at the end of the launch.
//
// WIDE = false (few registers): m and l are staged in `scratch` (2*n*G + 2*G
// floats of shared memory), then each thread sums one element at a time.
// WIDE = true: each thread owns E4 float4 groups of elements; every batch of
// U parts costs one round trip (O, m and l of all U parts loaded together)
// and folds into a running per-element max, as in the online softmax.
template <int G, int D, int NT, bool WIDE, class PartFn>
__device__ __forceinline__ void merge_parts(int n, PartFn part, __nv_bfloat16* out, float* dst, float* scratch,
                                            float2* stats = nullptr) {
  if constexpr (!WIDE) {
    float* wts = scratch;          // [n][G] m, then the weights
    float* ls = scratch + n * G;   // [n][G] l
    float* Ls = ls + n * G;        // [G]
    float* Ms = Ls + G;            // [G]
    for (int t = threadIdx.x; t < n * G; t += NT) {
      const float* pp = part(t / G) + G * D + (t % G);
      wts[t] = __ldcg(pp);
      ls[t] = __ldcg(pp + G);
    }
    named_barrier_sync(1, NT);
    if (threadIdx.x < G) {
      const int r = threadIdx.x;
      float M = -INFINITY;
      for (int j = 0; j < n; ++j) M = fmaxf(M, wts[j * G + r]);
      float L = 0.f;
      for (int j = 0; j < n; ++j) {
        const float mj = wts[j * G + r];
        const float w = (mj == -INFINITY) ? 0.f : fast_exp2(mj - M);
        wts[j * G + r] = w;
        L += w * ls[j * G + r];
      }
      Ls[r] = L;
      Ms[r] = M;
    }
    named_barrier_sync(1, NT);
    for (int idx = threadIdx.x; idx < G * D; idx += NT) {
      const int r = idx / D;
      float O = 0.f;
#pragma unroll 4
      for (int j = 0; j < n; ++j) O += wts[j * G + r] * __ldcg(part(j) + idx);
      if (out) {
        out[idx] = __float2bfloat16_rn(O / Ls[r]);
        if (stats && idx - r * D == 0) stats[r] = make_float2(Ms[r], Ls[r]);
      } else {
        __stcg(dst + idx, O);
        if (idx - r * D == 0) {
          __stcg(dst + G * D + r, Ms[r]);
          __stcg(dst + G * D + G + r, Ls[r]);
        }
      }
    }
  } else {
    constexpr int NV = G * D / 4;
    constexpr int E4 = (NV + NT - 1) / NT;
    constexpr int U = E4 <= 2 ? 8 : 4;
    float4 O[E4];
    float M[E4], L[E4];
    int vv[E4], rr[E4];
#pragma unroll
    for (int e = 0; e < E4; ++e) {
      O[e] = make_float4(0.f, 0.f, 0.f, 0.f);
      M[e] = -INFINITY;
      L[e] = 0.f;
      vv[e] = min((int)threadIdx.x + e * NT, NV - 1);
      rr[e] = vv[e] * 4 / D;
    }
    for (int j = 0; j < n; j += U) {
      float4 x[U][E4];
      float mj[U][E4], lj[U][E4];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const float* pp = part(min(j + u, n - 1));
#pragma unroll
        for (int e = 0; e < E4; ++e) {
          x[u][e] = __ldcg(reinterpret_cast<const float4*>(pp) + vv[e]);
          mj[u][e] = __ldcg(pp + G * D + rr[e]);
          lj[u][e] = __ldcg(pp + G * D + G + rr[e]);
        }
      }
#pragma unroll
      for (int e = 0; e < E4; ++e) {
        float bm = M[e];
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (j + u < n) bm = fmaxf(bm, mj[u][e]);
        const float sc = (M[e] == -INFINITY) ? 0.f : fast_exp2(M[e] - bm);
        O[e].x *= sc;
        O[e].y *= sc;
        O[e].z *= sc;
        O[e].w *= sc;
        L[e] *= sc;
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const float w = (j + u < n && mj[u][e] != -INFINITY) ? fast_exp2(mj[u][e] - bm) : 0.f;
          O[e].x += w * x[u][e].x;
          O[e].y += w * x[u][e].y;
          O[e].z += w * x[u][e].z;
          O[e].w += w * x[u][e].w;
          L[e] += w * lj[u][e];
        }
        M[e] = bm;
      }
    }
#pragma unroll
    for (int e = 0; e < E4; ++e) {
      const int v = threadIdx.x + e * NT;
      if (v >= NV) break;
      const int idx = v * 4, r = rr[e];
      if (out) {
        const float inv = 1.f / L[e];
        uint2 w;
        w.x = float2_to_bf16x2(O[e].x * inv, O[e].y * inv);
        w.y = float2_to_bf16x2(O[e].z * inv, O[e].w * inv);
        *reinterpret_cast<uint2*>(out + idx) = w;
        if (stats && idx - r * D == 0) stats[r] = make_float2(M[e], L[e]);
      } else {
        __stcg(reinterpret_cast<float4*>(dst + idx), O[e]);
        if (idx - r * D == 0) {
          __stcg(dst + G * D + r, M[e]);
          __stcg(dst + G * D + G + r, L[e]);
        }
      }
    }
  }
  named_barrier_sync(1, NT);
}

// After CTA p wrote its partial of item `id` (CTAs f..lst share it, f < lst),
// merge in two levels. Level 1: groups of kGroup consecutive CTAs; the last
// to arrive in a group merges the group into a group partial (slot 2 or 3 of
// the group's first CTA). Level 2: the last group to finish merges the group
// partials and writes the output. A one-group item writes the output at
// level 1. Run by the NT threads that wrote the partial; `flag` is one int
// of shared memory, `scratch` as for merge_parts.
template <int G, int D, int NT, bool WIDE>
__device__ __forceinline__ void merge_item(const DecodeArgs& a, int p, int f, int lst, int id,
                                           __nv_bfloat16* outp, float* scratch, volatile int* flag,
                                           float2* stats = nullptr) {
  // the barrier orders every thread's partial stores before thread 0's
  // counter update, whose release half publishes them; its acquire half
  // orders the other parts' stores before the loads below (the barrier
  // that follows carries that to the other threads). One acq_rel atomic
  // measured 2-4% faster per short step than a fence, a relaxed atomic and
  // a second fence.
  named_barrier_sync(1, NT);
  const int np = lst - f + 1;
  const int gi = (p - f) / kGroup, p0 = f + gi * kGroup;
  const int gsz = min(kGroup, lst - p0 + 1);
  const int n_groups = (np + kGroup - 1) / kGroup;
  const int gslot = (p0 == f) ? 1 : 0;  // the item is p0's last item iff p0 == f
  if (threadIdx.x == 0) {
    const uint32_t prev = atom_add_acq_rel_gpu(&a.gcounters[p0 * 2 + gslot], 1u);
    const bool last = prev == (uint32_t)(gsz - 1);
    if (last) a.gcounters[p0 * 2 + gslot] = 0u;
    *flag = last;
  }
  named_barrier_sync(1, NT);
  if (!*flag) return;
  auto own = [&](int j) {
    const int q = p0 + j;
    return partial_slot(a, q, q == f ? 1 : 0, G, D);
  };
  if (n_groups == 1) {
    merge_parts<G, D, NT, WIDE>(gsz, own, outp, nullptr, scratch, stats);
    return;
  }
  merge_parts<G, D, NT, WIDE>(gsz, own, nullptr, partial_slot(a, p0, 2 + gslot, G, D), scratch);
  if (threadIdx.x == 0) {
    const uint32_t prev = atom_add_acq_rel_gpu(&a.counters[id], 1u);
    const bool last = prev == (uint32_t)(n_groups - 1);
    if (last) a.counters[id] = 0u;
    *flag = last;
  }
  named_barrier_sync(1, NT);
  if (!*flag) return;
  auto grp_part = [&](int j) {
    const int q = f + j * kGroup;
    return partial_slot(a, q, 2 + (q == f ? 1 : 0), G, D);
  };
  merge_parts<G, D, NT, WIDE>(n_groups, grp_part, outp, nullptr, scratch, stats);
}

// The launch's last CTA advances every sequence length by one, except
// those of full sequences (seq_full), which it flags with kErrCapacity.
// Called by thread 0 after a __syncthreads that follows all of the CTA's
// work; `lens_s` is the kernel's shared-memory copy of the lengths (or
// null), which cannot have changed during the launch. A completed merge
// leaves its counters at zero; after a timeout some may be left behind, and
// a self-cleaning launch zeroes them and the error word. The launch's flags
// (timeout, capacity) are also ORed into the sticky status word when there
// is one; nothing in a launch clears it. Only a launch that reads its flags
// back (self-cleaning, or with a status word) needs its arrival to be an
// acquire-release atomic, which makes every CTA's error-word updates
// visible to the last one; otherwise the last CTA touches nothing another
// CTA wrote. Either way the next launch on the stream starts after this
// grid has completed, so nothing here needs a trailing fence.
__device__ __forceinline__ void finish_launch(const DecodeArgs& a, const int* lens_s) {
  const bool readback = a.self_clean || a.status != nullptr;
  const uint32_t prev = readback ? atom_add_acq_rel_gpu(a.done, 1u) : atomicAdd(a.done, 1u);
  if (prev == gridDim.x - 1) {
    bool full = false;
    for (int i = 0; i < a.geom.B; ++i) {
      const int t = lens_s ? lens_s[i] : a.lens[i];
      if (seq_full(a.geom, t))
        full = true;
      else
        a.lens[i] = t + 1;
    }
    if (readback) {
      const uint32_t e = *reinterpret_cast<volatile uint32_t*>(a.err);
      const uint32_t flags = e | (full ? kErrCapacity : 0u);
      if (a.status != nullptr && flags != 0u) atomicOr(a.status, flags);
      if (a.self_clean && e != 0u) {
        const int items = a.geom.B * (a.geom.n_r + a.geom.n_s);
        for (int i = 0; i < items; ++i) a.counters[i] = 0u;
        for (int i = 0; i < 2 * (int)gridDim.x; ++i) a.gcounters[i] = 0u;
        *a.err = 0u;
      }
      if (!a.self_clean && full) atomicOr(a.err, kErrCapacity);
    } else if (full) {
      atomicOr(a.err, kErrCapacity);
    }
    *a.done = 0u;
  }
}

}  // namespace dec
}  // namespace aoh
