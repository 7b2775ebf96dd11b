// H2Share anchor-layer selection (the paper's H2Share section and its GQA
// extension appendix): after an anchor decode step that wrote the scores of
// every retrieval row, each (sequence, retrieval KV head) keeps the top_k
// positions by group importance, the sum over the group's query heads of
// their attention probabilities. Ties go to the lower position; the
// positions are listed in increasing order, padded with -1 when fewer than
// top_k rows are held.
//
// The decode kernel leaves each retrieval head's final softmax state
// (M_h, L_h = sum of 2^(s - M_h), log2 units) beside the scores. One launch
// then does the rest, one thread-block cluster of kClus CTAs per item, CTA c
// owning the c-th contiguous slice of the item's rows, and warp w of a CTA
// the w-th contiguous run of its slice:
//   1. importance_j = sum_h 2^(s_hj - M_h) / L_h for the slice: the first
//      kSliceCap rows stay in shared memory, the rest go to a global
//      overflow buffer (read back from L2). The top 11 bits of every
//      importance are counted into a local histogram (importance is >= 0, so
//      its bit pattern orders like its value).
//   2. The bucket of those 11 bits that holds the top_k-th largest value:
//      every CTA adds its nonzero bins into CTA 0's histogram with remote
//      shared-memory atomics; one warp of CTA 0 picks the bucket and sends
//      (digit, rank) back.
//   3. Each warp lists the rows of its run at or above that bucket,
//      (position, bits) in position order, and counts those above it; the
//      listed rows not above it are the bucket's members (few, as a rule),
//      which go to CTA 0. CTA 0 finds the exact threshold among them (two
//      more radix levels, 11 and 10 bits), the number of rows equal to it
//      still needed, and from these every warp's output offset and share of
//      the equal rows, and sends each warp its plan. If some CTA has more
//      members than CTA 0 has room for, every level is instead a full pass
//      over the slices, as in step 2, followed by an exchange of per-CTA
//      counts.
//   4. Each warp writes its selected rows from its list: the rows above the
//      threshold and, in position order, as many rows equal to it as its
//      share (ballots give each row its place). A warp whose list
//      overflowed walks its run again, 128 rows at a time.
#include <stdint.h>

#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

constexpr int kClus = 8;              // CTAs per item (one cluster)
constexpr int kTopThreads = 512;
constexpr int kWarps = kTopThreads / 32;
constexpr int kBins = 2048;           // 11-bit digits
constexpr int kSliceCap = 18432;      // importance rows kept in shared memory per CTA (a multiple of 4)
constexpr int kCandC = 224;           // bucket members each CTA may send to CTA 0
constexpr int kKeepW = 128;           // rows at or above the bucket listed per warp
// CTA 0's region: first its level totals, later the cluster's members
// (bits, warp index)
constexpr int kRegion = kClus * kCandC * 8 > kBins * 4 ? kClus * kCandC * 8 : kBins * 4;
// slice, local histogram, region, per-warp lists of (position, bits)
constexpr int kTopSmem = kSliceCap * 4 + kBins * 4 + kRegion + kWarps * kKeepW * 8;
static_assert(kClus * kWarps == 128, "CTA 0 plans four warps per lane");
static_assert(kRegion % 16 == 0, "16-byte aligned list region");

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of `p`'s counterpart in the shared memory of cluster CTA `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
  return a;
}
__device__ __forceinline__ void cluster_red_add(uint32_t addr, uint32_t v) {
  asm volatile("red.relaxed.cluster.shared::cluster.add.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ void cluster_st(uint32_t addr, uint32_t x) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(x) : "memory");
}
__device__ __forceinline__ void cluster_st2(uint32_t addr, uint32_t x, uint32_t y) {
  asm volatile("st.shared::cluster.v2.u32 [%0], {%1, %2};" ::"r"(addr), "r"(x), "r"(y) : "memory");
}
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_sync() {
  cluster_arrive();
  cluster_wait();
}

__device__ __forceinline__ int warp_inclusive_scan(int v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += y;
  }
  return v;
}
// Run by one full warp: the digit, counted from the top of a kBins-bin
// histogram, whose bucket holds the r-th largest value (1 <= r <= total),
// and the rank within that bucket. First lane l sums the 64 digits
// kBins-64(l+1) .. kBins-1-64l and the block holding the rank is found;
// then lane l takes that block's digits 63-2l and 62-2l.
__device__ uint2 top_bucket_warp(const uint32_t* h, int r) {
  const int lane = threadIdx.x & 31;
  const uint32_t* hb = h + kBins - 64 * (lane + 1);
  int mine = 0;
#pragma unroll 4
  for (int i = 0; i < 64; i += 4) {
    const uint4 q = *reinterpret_cast<const uint4*>(hb + i);
    mine += (int)(q.x + q.y + q.z + q.w);
  }
  int inc = warp_inclusive_scan(mine);
  unsigned hit = __ballot_sync(0xffffffffu, inc - mine < r && inc >= r);
  int src = hit ? __ffs(hit) - 1 : 0;
  const int base = kBins - 64 * (src + 1);
  r -= __shfl_sync(0xffffffffu, inc - mine, src);
  const uint2 q = *reinterpret_cast<const uint2*>(h + base + 62 - 2 * lane);  // digits 62-2l, 63-2l of the block
  mine = (int)(q.x + q.y);
  inc = warp_inclusive_scan(mine);
  const int before = inc - mine;
  hit = __ballot_sync(0xffffffffu, before < r && inc >= r);
  src = hit ? __ffs(hit) - 1 : 0;
  const bool upper = r - before <= (int)q.y;  // the higher digit first
  const uint32_t d = (uint32_t)(base + 63 - 2 * lane - (upper ? 0 : 1));
  const uint32_t rr = (uint32_t)(upper ? r - before : r - before - (int)q.y);
  return make_uint2(__shfl_sync(0xffffffffu, d, src), __shfl_sync(0xffffffffu, rr, src));
}

// One radix level over the whole cluster: the local histogram `loc` is
// complete; add its nonzero bins into CTA 0's `tot`, let warp 0 of CTA 0 pick
// the bucket, zero `tot` again, and hand (digit, rank) to every CTA through
// `res`. Every thread of the cluster calls this.
__device__ uint32_t cluster_level(const uint32_t* loc, uint32_t* tot, uint2* res, int* rank, uint32_t crank) {
  for (int i = threadIdx.x; i < kBins; i += kTopThreads)
    if (loc[i]) cluster_red_add(cluster_addr(&tot[i], 0), loc[i]);
  cluster_sync();
  if (crank == 0 && threadIdx.x < 32) {
    const uint2 dr = top_bucket_warp(tot, *rank);
    for (int i = threadIdx.x * 4; i < kBins; i += 128) *reinterpret_cast<uint4*>(tot + i) = make_uint4(0, 0, 0, 0);
    if (threadIdx.x < kClus) cluster_st2(cluster_addr(res, threadIdx.x), dr.x, dr.y);
  }
  cluster_sync();
  *rank = (int)res->y;
  return res->x;
}

// The bucket of the CTA-local histogram h holding the rank-th largest value
// (every thread of the CTA calls this); *rank becomes the rank within it.
__device__ uint32_t cta_search(const uint32_t* h, int* rank, uint2* res) {
  if (threadIdx.x < 32) {
    const uint2 dr = top_bucket_warp(h, *rank);
    if (threadIdx.x == 0) *res = dr;
  }
  __syncthreads();
  const uint2 dr = *res;
  __syncthreads();  // h and res may be rewritten next
  *rank = (int)dr.y;
  return dr.x;
}

// Importance bits of slice rows r..r+3 (r a multiple of 4; past kSliceCap
// the rows live in the 16-byte aligned overflow buffer). Rows at or past
// `rows` are not meaningful: callers mask them.
__device__ __forceinline__ uint4 imp4(const float* s_imp, const float* over, int r, int rows) {
  if (r < kSliceCap) return *reinterpret_cast<const uint4*>(s_imp + r);
  if (r + 3 < rows) return __ldcg(reinterpret_cast<const uint4*>(over + r));
  uint4 x;
  x.x = r + 0 < rows ? __float_as_uint(__ldcg(over + r + 0)) : 0u;
  x.y = r + 1 < rows ? __float_as_uint(__ldcg(over + r + 1)) : 0u;
  x.z = r + 2 < rows ? __float_as_uint(__ldcg(over + r + 2)) : 0u;
  x.w = 0u;
  return x;
}
__device__ __forceinline__ uint32_t lane_of(const uint4& x, int i) {
  return i == 0 ? x.x : i == 1 ? x.y : i == 2 ? x.z : x.w;
}

// Exclusive prefix over the warp's lanes of a count in 0..4, and its total.
__device__ __forceinline__ int warp_scan4(int c, unsigned below, int* total) {
  int ex = 0, tot = 0;
#pragma unroll
  for (int k = 1; k <= 4; ++k) {
    const unsigned m = __ballot_sync(0xffffffffu, c >= k);
    ex += __popc(m & below);
    tot += __popc(m);
  }
  *total = tot;
  return ex;
}

// `stride` (the score and overflow row stride) is a multiple of 4, so every
// four-row group of scores or of overflow importances is one aligned 16-byte
// access.
template <int G>
__global__ void __cluster_dims__(kClus, 1, 1) __launch_bounds__(kTopThreads, 2)
    h2_topk_kernel(const float* scores, int stride, const int32_t* lens, int n_r, const float2* stats,
                   float* imp_over, int top_k, int32_t* idx_all) {
  extern __shared__ __align__(16) uint8_t dsm[];
  float* s_imp = reinterpret_cast<float*>(dsm);
  uint32_t* loc = reinterpret_cast<uint32_t*>(dsm + kSliceCap * 4);
  uint32_t* tot = loc + kBins;  // CTA 0: level totals, later the members
  const uint2* mem = reinterpret_cast<const uint2*>(tot);  // (bits, warp index)
  uint2* keep_all = reinterpret_cast<uint2*>(dsm + kSliceCap * 4 + kBins * 4 + kRegion);
  __shared__ float Mh[16], Linv[16];
  __shared__ int w_gt[kWarps], w_eq[kWarps];
  __shared__ uint2 res, lres;
  __shared__ int2 cnt[kClus];
  __shared__ int c_n[kClus];             // CTA 0: members each CTA found
  __shared__ int c_gt1[kClus * kWarps];  // CTA 0: rows above the bucket, per warp of the cluster
  __shared__ uint2 plan;                 // from CTA 0: (threshold, 1 if every level takes full passes)
  __shared__ int2 w_plan[kWarps];        // from CTA 0: (output offset, equal rows to take) per warp
  const uint32_t crank = cluster_rank();
  const int item = blockIdx.x / kClus, b = item / n_r;
  const int n = __ldcg(&lens[b]);
  int32_t* out = idx_all + (size_t)item * top_k;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const unsigned below = (1u << lane) - 1u;
  if (n <= top_k) {  // uniform over the cluster: every row is kept
    if (crank == 0)
      for (int j = t; j < top_k; j += kTopThreads) out[j] = j < n ? j : -1;
    return;
  }
  const int R = ((n + kClus - 1) / kClus + 31) & ~31;
  const int j0 = min(n, (int)crank * R), rows = min(n, j0 + R) - j0;
  float* over = imp_over + (size_t)item * stride + j0;  // indexed by slice row, used from kSliceCap on
  for (int i = t * 4; i < 2 * kBins; i += 4 * kTopThreads) *reinterpret_cast<uint4*>(loc + i) = make_uint4(0, 0, 0, 0);
  if (t < G) {
    const float2 st = __ldcg(&stats[(size_t)item * G + t]);
    Mh[t] = st.x;
    Linv[t] = 1.f / st.y;
  }
  __syncthreads();
  // CTA 0's totals are zero before any CTA adds into them
  cluster_arrive();

  // 1. importance of the slice, four rows per thread and step with every
  // score load of the step (heads in batches of at most 8) issued first
  constexpr int HB = G < 8 ? G : 8;
  const float* sc = scores + (size_t)item * G * stride + j0;
  for (int r = t * 4; r < rows; r += 4 * kTopThreads) {
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int h0 = 0; h0 < G; h0 += HB) {
      float4 sv[HB];
#pragma unroll
      for (int h = 0; h < HB; ++h) sv[h] = __ldcg(reinterpret_cast<const float4*>(sc + (size_t)(h0 + h) * stride + r));
#pragma unroll
      for (int h = 0; h < HB; ++h) {
        const float m = Mh[h0 + h], li = Linv[h0 + h];
        v.x += fast_exp2(sv[h].x - m) * li;
        v.y += fast_exp2(sv[h].y - m) * li;
        v.z += fast_exp2(sv[h].z - m) * li;
        v.w += fast_exp2(sv[h].w - m) * li;
      }
    }
    if (r < kSliceCap) {
      *reinterpret_cast<float4*>(s_imp + r) = v;
    } else if (r + 3 < rows) {
      __stcg(reinterpret_cast<float4*>(over + r), v);
    } else {
      over[r] = v.x;
      if (r + 1 < rows) over[r + 1] = v.y;
      if (r + 2 < rows) over[r + 2] = v.z;
    }
    // plain shared atomics (aggregating across the warp with a match costs
    // more than the conflicts it saves); four rows in one bin take one
    const uint32_t b0 = __float_as_uint(v.x) >> 21, b1 = __float_as_uint(v.y) >> 21;
    const uint32_t b2 = __float_as_uint(v.z) >> 21, b3 = __float_as_uint(v.w) >> 21;
    if (r + 3 < rows && b0 == b1 && b0 == b2 && b0 == b3) {
      atomicAdd(&loc[b0], 4u);
    } else {
      atomicAdd(&loc[b0], 1u);
      if (r + 1 < rows) atomicAdd(&loc[b1], 1u);
      if (r + 2 < rows) atomicAdd(&loc[b2], 1u);
      if (r + 3 < rows) atomicAdd(&loc[b3], 1u);
    }
  }
  __syncthreads();
  cluster_wait();

  // 2. the bucket of the top 11 bits holding the top_k-th largest value
  int rank = top_k;
  const uint32_t d1 = cluster_level(loc, tot, &res, &rank, crank);

  // 3. warp w owns slice rows [w*seg, (w+1)*seg), seg a multiple of 4, read
  // 128 at a time (rows 4*lane .. 4*lane+3, the next step's loads issued
  // before this step's rows are used). Each warp counts its rows above the
  // bucket and sends the bucket's members to CTA 0.
  const int seg = (((rows + kWarps - 1) / kWarps) + 3) & ~3;
  const int w0 = min(rows, warp * seg), w1 = min(rows, w0 + seg);
  uint2* keep = keep_all + warp * kKeepW;
  int nkeep = 0;  // rows at or above the bucket in this warp's run (listed while below kKeepW)
  {
    int gt1 = 0;
    // w0 is a multiple of 4 unless the run is empty (w0 == w1 == rows)
    uint4 xn = w0 < w1 ? imp4(s_imp, over, w0 + 4 * lane, rows) : make_uint4(0, 0, 0, 0);
    for (int rb = w0; rb < w1; rb += 128) {
      const uint4 x = xn;
      xn = imp4(s_imp, over, rb + 128 + 4 * lane, rows);
      const int r = rb + 4 * lane;
      uint32_t hi = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const bool in = r + i < w1;
        const uint32_t top = lane_of(x, i) >> 21;
        gt1 += in && top > d1;
        hi |= (uint32_t)(in && top >= d1) << i;
      }
      if (__any_sync(0xffffffffu, hi != 0)) {
        // the warp's list of candidate output rows, in position order
        int total;
        int k = nkeep + warp_scan4(__popc(hi), below, &total);
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if ((hi >> i) & 1u) {
            if (k < kKeepW) keep[k] = make_uint2((uint32_t)(j0 + r + i), lane_of(x, i));
            ++k;
          }
        nkeep += total;
      }
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) gt1 += __shfl_xor_sync(0xffffffffu, gt1, o);
    if (lane == 0) {
      cluster_st(cluster_addr(&c_gt1[crank * kWarps + warp], 0), (uint32_t)gt1);
      // the bucket's members are the listed rows not above it; a warp whose
      // list is incomplete cannot send them (kCandC + 1 marks the CTA full)
      w_eq[warp] = nkeep <= kKeepW ? nkeep - gt1 : kCandC + 1;
    }
    __syncthreads();
    int off = 0, n_cta = 0;
    for (int w = 0; w < kWarps; ++w) {
      if (w < warp) off += w_eq[w];
      n_cta += w_eq[w];
    }
    if (n_cta <= kCandC) {
      // send this warp's members to CTA 0, at offset `off` of this CTA's part
      const uint32_t mem_dst = cluster_addr(mem + crank * kCandC, 0);
      for (int c0 = 0; c0 < nkeep; c0 += 32) {
        const int c = c0 + lane;
        const uint2 e = c < nkeep ? keep[c] : make_uint2(0u, 0u);
        const bool is_mem = c < nkeep && (e.y >> 21) == d1;
        const unsigned mm = __ballot_sync(0xffffffffu, is_mem);
        if (is_mem) cluster_st2(mem_dst + 8u * (uint32_t)(off + __popc(mm & below)), e.y, (uint32_t)warp);
        off += __popc(mm);
      }
    }
    if (t == 0) cluster_st(cluster_addr(&c_n[crank], 0), (uint32_t)min(n_cta, kCandC + 1));
  }
  cluster_sync();  // CTA 0 holds the cluster's members and counts

  if (crank == 0) {
    bool full = false;
    for (int c = 0; c < kClus; ++c) full |= c_n[c] > kCandC;
    if (!full) {
      // the last two levels over the members alone
      uint32_t prefix = d1 << 21, mask = 0xFFE00000u;
      int rk = rank;
#pragma unroll 1
      for (int level = 1; level < 3; ++level) {
        const int sh = level == 1 ? 10 : 0;
        const uint32_t dmask = level == 1 ? 0x7FFu : 0x3FFu;
        for (int i = t * 4; i < kBins; i += 4 * kTopThreads) *reinterpret_cast<uint4*>(loc + i) = make_uint4(0, 0, 0, 0);
        __syncthreads();
        for (int s = t; s < kClus * kCandC; s += kTopThreads) {
          if (s % kCandC >= c_n[s / kCandC]) continue;
          const uint32_t bits = mem[s].x;
          if ((bits & mask) == prefix) atomicAdd(&loc[(bits >> sh) & dmask], 1u);
        }
        __syncthreads();
        prefix |= cta_search(loc, &rk, &lres) << sh;
        mask |= dmask << sh;
      }
      const uint32_t thr = prefix;
      const int need_eq = rk;
      // per warp of the cluster: members above the threshold and equal to it
      if (t < 2 * kClus * kWarps) loc[t] = 0u;
      __syncthreads();
      for (int s = t; s < kClus * kCandC; s += kTopThreads) {
        const int c = s / kCandC;
        if (s % kCandC >= c_n[c]) continue;
        const uint2 m = mem[s];
        const uint32_t bits = m.x;
        const int gw = c * kWarps + (int)m.y;
        if (bits > thr)
          atomicAdd(&loc[gw], 1u);
        else if (bits == thr)
          atomicAdd(&loc[kClus * kWarps + gw], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        // lane l plans warps 4l .. 4l+3 of the cluster (position order);
        // equal rows go to the lowest positions first
        constexpr int NW = kClus * kWarps;
        int gtv[4], eqv[4], eqs = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int g = 4 * lane + q;
          gtv[q] = c_gt1[g] + (int)loc[g];
          eqv[q] = (int)loc[NW + g];
          eqs += eqv[q];
        }
        int eq_run = warp_inclusive_scan(eqs) - eqs;
        int tk[4], ks = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          tk[q] = max(0, min(eqv[q], need_eq - eq_run));
          eq_run += eqv[q];
          ks += gtv[q] + tk[q];
        }
        int k_run = warp_inclusive_scan(ks) - ks;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int g = 4 * lane + q;
          cluster_st2(cluster_addr(&w_plan[g % kWarps], (uint32_t)(g / kWarps)), (uint32_t)k_run, (uint32_t)tk[q]);
          k_run += gtv[q] + tk[q];
        }
        if (lane < kClus) cluster_st2(cluster_addr(&plan, (uint32_t)lane), thr, 0u);
      }
    } else {
      // too many members: zero the totals for full passes
      for (int i = t * 4; i < kBins; i += 4 * kTopThreads) *reinterpret_cast<uint4*>(tot + i) = make_uint4(0, 0, 0, 0);
      if (t < kClus) cluster_st2(cluster_addr(&plan, (uint32_t)t), 0u, 1u);
    }
  }
  cluster_sync();  // every CTA holds its plan

  uint32_t thr;
  int pos, take_eq;
  if (plan.y == 0u) {
    thr = plan.x;
    pos = w_plan[warp].x;
    take_eq = w_plan[warp].y;
  } else {
    // full passes: levels 2 and 3 over every slice, then per-CTA counts
    uint32_t prefix = d1 << 21, mask = 0xFFE00000u;
#pragma unroll 1
    for (int level = 1; level < 3; ++level) {
      const int sh = level == 1 ? 10 : 0;
      const uint32_t dmask = level == 1 ? 0x7FFu : 0x3FFu;
      for (int i = t * 4; i < kBins; i += 4 * kTopThreads) *reinterpret_cast<uint4*>(loc + i) = make_uint4(0, 0, 0, 0);
      __syncthreads();
      for (int r = t * 4; r < rows; r += 4 * kTopThreads) {
        const uint4 x = imp4(s_imp, over, r, rows);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t bits = lane_of(x, i);
          if (r + i < rows && (bits & mask) == prefix) atomicAdd(&loc[(bits >> sh) & dmask], 1u);
        }
      }
      __syncthreads();
      prefix |= cluster_level(loc, tot, &res, &rank, crank) << sh;
      mask |= dmask << sh;
    }
    thr = prefix;
    const int need_eq = rank;
    int gt = 0, eq = 0;
    for (int rb = w0; rb < w1; rb += 128) {
      const int r = rb + 4 * lane;
      const uint4 x = imp4(s_imp, over, r, rows);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t y = lane_of(x, i);
        gt += r + i < w1 && y > thr;
        eq += r + i < w1 && y == thr;
      }
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      gt += __shfl_xor_sync(0xffffffffu, gt, o);
      eq += __shfl_xor_sync(0xffffffffu, eq, o);
    }
    if (lane == 0) {
      w_gt[warp] = gt;
      w_eq[warp] = eq;
    }
    __syncthreads();
    int gt_cta = 0, eq_cta = 0, eq_before_w = 0;
    for (int w = 0; w < kWarps; ++w) {
      if (w < warp) eq_before_w += w_eq[w];
      gt_cta += w_gt[w];
      eq_cta += w_eq[w];
    }
    if (t < kClus) cluster_st2(cluster_addr(&cnt[crank], (uint32_t)t), (uint32_t)gt_cta, (uint32_t)eq_cta);
    cluster_sync();  // no shared memory of another CTA is touched after this
    // equal rows go to the lowest positions first: the CTAs before this one,
    // then the warps before this one, take theirs first
    pos = 0;
    int eq_run = 0;
    for (int c = 0; c < (int)crank; ++c) {
      const int2 x = cnt[c];
      pos += x.x + max(0, min(x.y, need_eq - eq_run));
      eq_run += x.y;
    }
    const int take_cta = max(0, min(eq_cta, need_eq - eq_run));
    int eq_w = 0;
    for (int w = 0; w < warp; ++w) {
      pos += w_gt[w] + max(0, min(w_eq[w], take_cta - eq_w));
      eq_w += w_eq[w];
    }
    take_eq = max(0, min(eq, take_cta - eq_before_w));
  }

  // 4. ordered compaction of the warp's run: from its list when the list
  // holds every row at or above the bucket (the threshold lies in it), else
  // by a pass over the run
  int taken = 0;  // equal rows met so far by this warp
  if (nkeep <= kKeepW) {
    for (int c0 = 0; c0 < nkeep; c0 += 32) {
      const int c = c0 + lane;
      const uint2 e = c < nkeep ? keep[c] : make_uint2(0u, 0u);
      const bool is_gt = c < nkeep && e.y > thr;
      const bool is_eq = c < nkeep && e.y == thr;
      const unsigned eqm = __ballot_sync(0xffffffffu, is_eq);
      const bool kp = is_gt || (is_eq && taken + __popc(eqm & below) < take_eq);
      const unsigned km = __ballot_sync(0xffffffffu, kp);
      const int p = pos + __popc(km & below);
      if (kp && p < top_k) out[p] = (int32_t)e.x;
      pos += __popc(km);
      taken += __popc(eqm);
    }
    return;
  }
  uint4 xn = w0 < w1 ? imp4(s_imp, over, w0 + 4 * lane, rows) : make_uint4(0, 0, 0, 0);
  for (int rb = w0; rb < w1; rb += 128) {
    const uint4 x = xn;
    xn = imp4(s_imp, over, rb + 128 + 4 * lane, rows);
    const int r = rb + 4 * lane;
    uint32_t keep = 0, eqb = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t y = lane_of(x, i);
      const bool in = r + i < w1;
      keep |= (uint32_t)(in && y > thr) << i;
      eqb |= (uint32_t)(in && y == thr) << i;
    }
    if (__any_sync(0xffffffffu, eqb != 0)) {
      // the equal rows of this step in position order: lanes before this one
      // first, then this lane's in row order
      int tot_eq;
      int e = taken + warp_scan4(__popc(eqb), below, &tot_eq);
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if ((eqb >> i) & 1u) {
          if (e < take_eq) keep |= 1u << i;
          ++e;
        }
      taken += tot_eq;
    }
    int tot_keep;
    int p = pos + warp_scan4(__popc(keep), below, &tot_keep);
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if ((keep >> i) & 1u) {
        if (p < top_k) out[p] = j0 + r + i;
        ++p;
      }
    pos += tot_keep;
  }
}

}  // namespace

// Every segment starts on a 16-byte boundary (the head states are float2,
// and max_seq may be odd).
inline size_t pad4(size_t n) { return (n + 3) / 4 * 4; }

// Rows of scores and of the overflow buffer are padded to a multiple of 4
// floats (16-byte loads of four rows).
inline int score_stride(int max_seq) { return (int)pad4((size_t)max_seq); }

// Importance rows spill to global memory only past kSliceCap rows of a
// cluster CTA's slice, that is for sequences longer than kClus * kSliceCap.
inline size_t overflow_floats(size_t items, int max_seq) {
  return max_seq > kClus * kSliceCap ? items * (size_t)score_stride(max_seq) : 0;
}

size_t h2_workspace_floats(int B, int n_r, int G, int max_seq) {
  const size_t items = (size_t)B * n_r;
  // scores, per-head (max, sum) states (float2), importance overflow
  return items * G * (size_t)score_stride(max_seq) + pad4(items * G * 2) + overflow_floats(items, max_seq);
}

namespace {
struct H2Layout {
  float* scores;
  float2* stats;
  float* imp_over;
};
H2Layout h2_layout(float* ws, int B, int n_r, int G, int max_seq) {
  const size_t items = (size_t)B * n_r;
  H2Layout l;
  l.scores = ws;
  l.stats = reinterpret_cast<float2*>(l.scores + items * G * (size_t)score_stride(max_seq));
  l.imp_over = reinterpret_cast<float*>(l.stats) + pad4(items * G * 2);
  return l;
}

template <int G>
cudaError_t launch_topk_g(const H2Layout& l, int max_seq, const int32_t* lens, int n_r, int top_k, int32_t* idx_out,
                          unsigned grid, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    const cudaError_t e = cudaFuncSetAttribute(h2_topk_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTopSmem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  h2_topk_kernel<G><<<grid, kTopThreads, kTopSmem, s>>>(l.scores, score_stride(max_seq), lens, n_r, l.stats,
                                                         l.imp_over, top_k, idx_out);
  return cudaGetLastError();
}
}  // namespace

void h2_decode_outputs(float* ws, int B, int n_r, int G, int max_seq, float** scores, int* stride, float2** stats) {
  const H2Layout l = h2_layout(ws, B, n_r, G, max_seq);
  *scores = l.scores;
  *stride = score_stride(max_seq);
  *stats = l.stats;
}

cudaError_t launch_h2_topk(float* ws, int max_seq, const int32_t* lens, int B, int n_r, int G, int top_k,
                           int32_t* idx_out, cudaStream_t s) {
  if (B * n_r == 0) return cudaSuccess;
  const size_t items = (size_t)B * n_r;
  if (items * kClus > 0x7fffffffu) return cudaErrorInvalidValue;
  const H2Layout l = h2_layout(ws, B, n_r, G, max_seq);
  const unsigned grid = (unsigned)(items * kClus);
  switch (G) {
#define AOH_TOPK(g) \
  case g:           \
    return launch_topk_g<g>(l, max_seq, lens, n_r, top_k, idx_out, grid, s);
    AOH_TOPK(1) AOH_TOPK(2) AOH_TOPK(3) AOH_TOPK(4) AOH_TOPK(5) AOH_TOPK(6) AOH_TOPK(7) AOH_TOPK(8) AOH_TOPK(16)
#undef AOH_TOPK
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace aoh
