// Split-KV flash-decode for head-heterogeneous attention (Sec. 5, "Decode
// Stage", Eq. 8): one new token per sequence; retrieval KV heads attend over
// their whole history, streaming KV heads over their S sink + W window slots.
//
// One CTA = one (sequence b, KV head, split) work unit; a split is a
// contiguous range of cache rows. All G query heads of the GQA group are
// processed against each K/V row, so every cached byte is read from HBM once.
//
//   warp NW (producer): cp.async.bulk (TMA) copies of K and V row tiles into
//     an NST-stage shared-memory ring guarded by full/empty mbarriers. The
//     new token's K/V row is copied from the input in place of its cache row,
//     and the same warp appends it to the cache (retrieval row t, or ring slot
//     S + (t - S) mod W for a streaming head).
//   warps 0..NW-1 (consumers): lanes are split into groups of LPT = D/8 lanes;
//     each lane owns 8 consecutive d-elements of a row. A group takes NT rows
//     of a tile, forms partial q.k dot products for all G heads with packed
//     f32x2 FMAs, finishes them with a butterfly reduce-scatter of shuffles,
//     and keeps the online-softmax state (running max m, sum l, output o) in
//     registers. The running max is only moved when a new score exceeds it by
//     more than 2^8 (the result is unchanged: numerator and denominator use
//     the same offset).
//   end of CTA: groups merge through shared memory; a single split writes the
//     bf16 output, several splits write fp32 partials and the last CTA to
//     arrive at the (b, head) counter merges them (log-sum-exp weights). The
//     last CTA of the launch advances every sequence length by one.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

using bf16 = __nv_bfloat16;
constexpr unsigned kFull = 0xffffffffu;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D_, int G_>
struct DecodeCfg {
  static constexpr int D = D_;
  static constexpr int G = G_;
  static constexpr int LPT = D / 8;              // lanes per token group
  static constexpr int GPW = 32 / LPT;           // groups per warp
  static constexpr int GP = cmax(2, next_pow2(G));  // rows padded to a power of two (>= 2)
  static constexpr int NT = cmax(4, LPT / GP);   // rows per group per tile
  static constexpr int V = NT * GP;              // partial dots per lane
  static constexpr int RP = V / LPT;             // values per lane after reduce-scatter
  static constexpr int Q = GP / RP;              // lanes holding distinct row sets
  static constexpr int NW = 4;                   // consumer warps
  static constexpr int NG = NW * GPW;            // groups per CTA
  static constexpr int TOK = NG * NT;            // rows per tile
  static constexpr int RB = D * 2;               // bytes per row
  static constexpr int NST = 6;                  // pipeline stages
  static constexpr int STAGE_BYTES = TOK * RB * 2;
  static constexpr int DATA_BYTES = NST * STAGE_BYTES;
  static constexpr int MERGE_BYTES = NG * G * (D + 2) * 4;
  static constexpr int COMBINE_BYTES = kMaxSplits * G * 4 + 2 * G * 4;
  static constexpr int SMEM = DATA_BYTES + 2 * NST * 8 + 16;
  static constexpr int THREADS = (NW + 1) * 32;
  static_assert(V % LPT == 0 && RP <= GP, "bad reduce-scatter shape");
  static_assert(MERGE_BYTES <= DATA_BYTES && COMBINE_BYTES <= DATA_BYTES, "merge area");
};

// Copy rows [row0, row0 + cnt) of one region into shared memory; row xr (if
// inside the range) comes from the new token instead of the cache.
template <int RB>
__device__ __forceinline__ void copy_rows(uint8_t* dst, const uint8_t* rows, const uint8_t* new_row, int row0,
                                          int cnt, int xr, uint64_t* bar) {
  const int row1 = row0 + cnt;
  if (xr >= row0 && xr < row1) {
    if (xr > row0) bulk_g2s(dst, rows + (size_t)row0 * RB, (uint32_t)(xr - row0) * RB, bar);
    bulk_g2s(dst + (size_t)(xr - row0) * RB, new_row, RB, bar);
    if (row1 > xr + 1)
      bulk_g2s(dst + (size_t)(xr + 1 - row0) * RB, rows + (size_t)(xr + 1) * RB, (uint32_t)(row1 - xr - 1) * RB,
               bar);
  } else {
    bulk_g2s(dst, rows + (size_t)row0 * RB, (uint32_t)cnt * RB, bar);
  }
}

// Butterfly reduce-scatter over the LPT lanes of a group: on return lane c
// holds in x[0..RP) the group sums of values [c*RP, (c+1)*RP).
template <int LPT, int V>
__device__ __forceinline__ void reduce_scatter(float (&x)[V], int c) {
  int n = V;
#pragma unroll
  for (int m = LPT / 2; m >= 1; m /= 2) {
    const int half = n / 2;
    const bool up = (c & m) != 0;
#pragma unroll
    for (int k = 0; k < V / 2; ++k) {
      if (k < half) {
        const float lo = x[k], hi = x[k + half];
        const float send = up ? lo : hi;
        const float keep = up ? hi : lo;
        x[k] = keep + __shfl_xor_sync(kFull, send, m);
      }
    }
    n = half;
  }
}

template <class C>
__global__ void __launch_bounds__(C::THREADS) decode_kernel(const __grid_constant__ DecodeArgs a) {
  constexpr int D = C::D, G = C::G, RB = C::RB, TOK = C::TOK, NST = C::NST;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::DATA_BYTES);
  uint64_t* empty = full + NST;
  int* flag = reinterpret_cast<int*>(empty + NST);

  const CacheGeom& g = a.geom;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // ---- work unit
  const int per_b = g.n_r * a.ns_r + g.n_s * a.ns_s;
  const int b = blockIdx.x / per_b;
  int rem = blockIdx.x - b * per_b;
  int kind, hi, split, nsplit;
  if (rem < g.n_r * a.ns_r) {
    kind = 0; hi = rem / a.ns_r; split = rem - hi * a.ns_r; nsplit = a.ns_r;
  } else {
    rem -= g.n_r * a.ns_r;
    kind = 1; hi = rem / a.ns_s; split = rem - hi * a.ns_s; nsplit = a.ns_s;
  }
  const int kvh = kind ? g.s_head[hi] : g.r_head[hi];
  const int t = __ldcg(&a.lens[b]);  // position of the new token
  int n, xr, cap;
  if (kind == 0) {
    cap = g.max_seq; n = t + 1; xr = t;
  } else {
    cap = g.S + g.W; n = min(t + 1, cap); xr = t < g.S ? t : g.S + (t - g.S) % g.W;
  }
  const int chunk = (n + nsplit - 1) / nsplit;
  const int r_begin = min(n, split * chunk);
  const int r_end = min(n, r_begin + chunk);
  const int n_tiles = (r_end - r_begin + TOK - 1) / TOK;

  const size_t reg = kind ? g.s_region(b, hi) : g.r_region(b, hi);
  const uint8_t* Kc = reinterpret_cast<const uint8_t*>(static_cast<const bf16*>(a.kv) + reg);
  const uint8_t* Vc = Kc + (size_t)cap * RB;
  const size_t new_off = ((size_t)b * g.Hkv + kvh) * D;
  const uint8_t* kn = reinterpret_cast<const uint8_t*>(static_cast<const bf16*>(a.k_new) + new_off);
  const uint8_t* vn = reinterpret_cast<const uint8_t*>(static_cast<const bf16*>(a.v_new) + new_off);

  if (threadIdx.x == 0) {
#pragma unroll
    for (int s = 0; s < NST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], C::NW);
    }
    fence_mbar_init();
  }
  __syncthreads();

  float m[G], l[G];
  float2 o[G][4];
  const int gi = lane / C::LPT, c = lane % C::LPT;
  const int grp = warp * C::GPW + gi;

  if (warp == C::NW) {
    // ------------------------------------------------------------ producer
    if (xr >= r_begin && xr < r_end && lane < D / 8) {
      uint8_t* Kw = const_cast<uint8_t*>(Kc);
      uint8_t* Vw = const_cast<uint8_t*>(Vc);
      reinterpret_cast<uint4*>(Kw + (size_t)xr * RB)[lane] = reinterpret_cast<const uint4*>(kn)[lane];
      reinterpret_cast<uint4*>(Vw + (size_t)xr * RB)[lane] = reinterpret_cast<const uint4*>(vn)[lane];
    }
    if (lane == 0) {
      int issued = 0;
      for (int it = 0; it < n_tiles; ++it) {
        const int st = it % NST;
        const uint32_t ph = (it / NST) & 1;
        if (it >= NST && !mbar_wait(&empty[st], ph ^ 1, a.err)) break;
        const int row0 = r_begin + it * TOK;
        const int cnt = min(TOK, r_end - row0);
        mbar_arrive_expect_tx(&full[st], (uint32_t)cnt * RB * 2);
        uint8_t* ks = smem + st * C::STAGE_BYTES;
        copy_rows<RB>(ks, Kc, kn, row0, cnt, xr, &full[st]);
        copy_rows<RB>(ks + TOK * RB, Vc, vn, row0, cnt, xr, &full[st]);
        issued = it + 1;
      }
      // Every issued copy has landed before shared memory is reused (normally
      // the consumers already waited for all of them).
      for (int it = issued > NST ? issued - NST : 0; it < issued; ++it)
        mbar_wait(&full[it % NST], (it / NST) & 1, a.err);
    }
  } else {
    // ------------------------------------------------------------ consumers
    float2 qf[G][4];
    const bf16* qb = static_cast<const bf16*>(a.q) + ((size_t)b * g.Hq + (size_t)kvh * G) * D + c * 8;
#pragma unroll
    for (int r = 0; r < G; ++r) {
      const uint4 raw = *reinterpret_cast<const uint4*>(qb + (size_t)r * D);
      qf[r][0] = bf16x2_to_float2(raw.x);
      qf[r][1] = bf16x2_to_float2(raw.y);
      qf[r][2] = bf16x2_to_float2(raw.z);
      qf[r][3] = bf16x2_to_float2(raw.w);
      m[r] = -INFINITY;
      l[r] = 0.f;
#pragma unroll
      for (int e = 0; e < 4; ++e) o[r][e] = make_float2(0.f, 0.f);
    }
    const int tb = grp * C::NT;  // first tile row of this group

    for (int it = 0; it < n_tiles; ++it) {
      const int st = it % NST;
      const uint32_t ph = (it / NST) & 1;
      if (!mbar_wait(&full[st], ph, a.err)) break;
      const int cnt = min(TOK, r_end - (r_begin + it * TOK));
      const uint8_t* ks = smem + st * C::STAGE_BYTES;
      const uint8_t* vs = ks + TOK * RB;

      // partial q.k over this lane's 8 d-elements, for NT rows x G heads
      float part[C::V];
      {
        float2 kf[C::NT][4];
#pragma unroll
        for (int tt = 0; tt < C::NT; ++tt) {
          const int row = min(tb + tt, cnt - 1);
          const uint4 raw = lds128(ks + row * RB + c * 16);
          kf[tt][0] = bf16x2_to_float2(raw.x);
          kf[tt][1] = bf16x2_to_float2(raw.y);
          kf[tt][2] = bf16x2_to_float2(raw.z);
          kf[tt][3] = bf16x2_to_float2(raw.w);
        }
#pragma unroll
        for (int tt = 0; tt < C::NT; ++tt) {
#pragma unroll
          for (int r = 0; r < C::GP; ++r) {
            if (r < G) {
              float2 acc = make_float2(0.f, 0.f);
#pragma unroll
              for (int e = 0; e < 4; ++e) acc = __ffma2_rn(qf[r][e], kf[tt][e], acc);
              part[tt * C::GP + r] = acc.x + acc.y;
            } else {
              part[tt * C::GP + r] = 0.f;
            }
          }
        }
      }
      reduce_scatter<C::LPT, C::V>(part, c);

      // scores held by this lane: value v = c*RP + k -> row tt = v / GP, head r = v % GP
      float s[C::RP], mx[C::RP];
#pragma unroll
      for (int k = 0; k < C::RP; ++k) {
        const int v = c * C::RP + k;
        const int tt = v / C::GP, r = v % C::GP;
        const bool valid = (tb + tt < cnt) && (r < G);
        s[k] = valid ? part[k] * a.scale_log2 : -INFINITY;
        mx[k] = s[k];
      }
#pragma unroll
      for (int msk = C::Q; msk < C::LPT; msk *= 2)
#pragma unroll
        for (int k = 0; k < C::RP; ++k) mx[k] = fmaxf(mx[k], __shfl_xor_sync(kFull, mx[k], msk));
      float bm[G];
#pragma unroll
      for (int j = 0; j < C::Q; ++j)
#pragma unroll
        for (int k = 0; k < C::RP; ++k)
          if (j * C::RP + k < G) bm[j * C::RP + k] = __shfl_sync(kFull, mx[k], gi * C::LPT + j);

      bool need = false;
#pragma unroll
      for (int r = 0; r < G; ++r) need |= bm[r] > m[r] + kRescaleThreshold;
      if (__any_sync(kFull, need)) {
#pragma unroll
        for (int r = 0; r < G; ++r) {
          const float mn = fmaxf(m[r], bm[r]);
          const float alpha = (m[r] == -INFINITY) ? 0.f : fast_exp2(m[r] - mn);
          m[r] = mn;
          l[r] *= alpha;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            o[r][e].x *= alpha;
            o[r][e].y *= alpha;
          }
        }
      }

      float p[C::RP];
#pragma unroll
      for (int k = 0; k < C::RP; ++k) {
        const int r = (c % C::Q) * C::RP + k;
        float mr = m[0];
#pragma unroll
        for (int rr = 1; rr < G; ++rr) mr = (rr == r) ? m[rr] : mr;
        p[k] = (s[k] == -INFINITY) ? 0.f : fast_exp2(s[k] - mr);
      }

      float2 vf[C::NT][4];
#pragma unroll
      for (int tt = 0; tt < C::NT; ++tt) {
        const int row = min(tb + tt, cnt - 1);
        const uint4 raw = lds128(vs + row * RB + c * 16);
        vf[tt][0] = bf16x2_to_float2(raw.x);
        vf[tt][1] = bf16x2_to_float2(raw.y);
        vf[tt][2] = bf16x2_to_float2(raw.z);
        vf[tt][3] = bf16x2_to_float2(raw.w);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);

#pragma unroll
      for (int tt = 0; tt < C::NT; ++tt) {
#pragma unroll
        for (int r = 0; r < G; ++r) {
          const int v = tt * C::GP + r;
          const float pv = __shfl_sync(kFull, p[v % C::RP], gi * C::LPT + v / C::RP);
          l[r] += pv;
          const float2 pp = make_float2(pv, pv);
#pragma unroll
          for (int e = 0; e < 4; ++e) o[r][e] = __ffma2_rn(pp, vf[tt][e], o[r][e]);
        }
      }
    }
  }

  // ---- merge the groups of this CTA (stage memory is free now)
  __syncthreads();
  float* mo = reinterpret_cast<float*>(smem);           // [NG][G][D]
  float* mm = mo + C::NG * G * D;                        // [NG][G]
  float* ml = mm + C::NG * G;                            // [NG][G]
  if (warp < C::NW) {
#pragma unroll
    for (int r = 0; r < G; ++r) {
      float* dst = mo + ((size_t)grp * G + r) * D + c * 8;
#pragma unroll
      for (int e = 0; e < 4; ++e) *reinterpret_cast<float2*>(dst + 2 * e) = o[r][e];
      if (c == 0) {
        mm[grp * G + r] = m[r];
        ml[grp * G + r] = l[r];
      }
    }
  }
  __syncthreads();

  const bool single = nsplit == 1;
  float* part_base = a.partials + (((size_t)b * g.Hkv + kvh) * a.split_stride + split) * (size_t)(G * (D + 2));
  bf16* outp = static_cast<bf16*>(a.out) + ((size_t)b * g.Hq + (size_t)kvh * G) * D;
  for (int idx = threadIdx.x; idx < G * D; idx += C::THREADS) {
    const int r = idx / D, d = idx - r * D;
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < C::NG; ++q) M = fmaxf(M, mm[q * G + r]);
    float O = 0.f, L = 0.f;
#pragma unroll
    for (int q = 0; q < C::NG; ++q) {
      const float mq = mm[q * G + r];
      const float w = (mq == -INFINITY) ? 0.f : fast_exp2(mq - M);
      O += w * mo[((size_t)q * G + r) * D + d];
      L += w * ml[q * G + r];
    }
    if (single) {
      outp[idx] = __float2bfloat16_rn(O / L);
    } else {
      __stcg(part_base + idx, O);
      if (d == 0) {
        __stcg(part_base + G * D + r, M);
        __stcg(part_base + G * D + G + r, L);
      }
    }
  }

  if (!single) {
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      const uint32_t prev = atomicAdd(&a.counters[b * g.Hkv + kvh], 1u);
      *flag = (prev == (uint32_t)nsplit - 1u);
    }
    __syncthreads();
    if (*flag) {
      __threadfence();
      // last split to finish: merge all partials of (b, head)
      float* wts = reinterpret_cast<float*>(smem);  // [nsplit][G]
      float* Ls = wts + kMaxSplits * G;             // [G]
      const float* pb0 = a.partials + ((size_t)b * g.Hkv + kvh) * a.split_stride * (size_t)(G * (D + 2));
      if (threadIdx.x < G) {
        const int r = threadIdx.x;
        float M = -INFINITY;
        for (int sp = 0; sp < nsplit; ++sp) M = fmaxf(M, __ldcg(pb0 + (size_t)sp * G * (D + 2) + G * D + r));
        float L = 0.f;
        for (int sp = 0; sp < nsplit; ++sp) {
          const float* pb = pb0 + (size_t)sp * G * (D + 2);
          const float ms = __ldcg(pb + G * D + r);
          const float w = (ms == -INFINITY) ? 0.f : fast_exp2(ms - M);
          wts[sp * G + r] = w;
          L += w * __ldcg(pb + G * D + G + r);
        }
        Ls[r] = L;
      }
      __syncthreads();
      for (int idx = threadIdx.x; idx < G * D; idx += C::THREADS) {
        const int r = idx / D;
        float O = 0.f;
        for (int sp = 0; sp < nsplit; ++sp) O += wts[sp * G + r] * __ldcg(pb0 + (size_t)sp * G * (D + 2) + idx);
        outp[idx] = __float2bfloat16_rn(O / Ls[r]);
      }
      if (threadIdx.x == 0) a.counters[b * g.Hkv + kvh] = 0u;
    }
  }

  // ---- the launch's last CTA advances the lengths
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const uint32_t prev = atomicAdd(a.done, 1u);
    if (prev == gridDim.x - 1) {
      for (int i = 0; i < g.B; ++i) a.lens[i] += 1;
      __threadfence();
      *a.done = 0u;
    }
  }
}

template <int D, int G>
cudaError_t launch_cfg(const DecodeArgs& a, int n_ctas, cudaStream_t s) {
  using C = DecodeCfg<D, G>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  decode_kernel<C><<<n_ctas, C::THREADS, C::SMEM, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

bool decode_supported(int D, int G) {
  if (D != 64 && D != 128) return false;
  return G == 1 || G == 2 || G == 4 || G == 7 || G == 8;
}

cudaError_t launch_decode(const DecodeArgs& a, int n_ctas, cudaStream_t s) {
  const int D = a.geom.D, G = a.geom.G;
  if (D == 128) {
    switch (G) {
      case 1: return launch_cfg<128, 1>(a, n_ctas, s);
      case 2: return launch_cfg<128, 2>(a, n_ctas, s);
      case 4: return launch_cfg<128, 4>(a, n_ctas, s);
      case 7: return launch_cfg<128, 7>(a, n_ctas, s);
      case 8: return launch_cfg<128, 8>(a, n_ctas, s);
    }
  } else if (D == 64) {
    switch (G) {
      case 1: return launch_cfg<64, 1>(a, n_ctas, s);
      case 2: return launch_cfg<64, 2>(a, n_ctas, s);
      case 4: return launch_cfg<64, 4>(a, n_ctas, s);
      case 7: return launch_cfg<64, 7>(a, n_ctas, s);
      case 8: return launch_cfg<64, 8>(a, n_ctas, s);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace aoh
