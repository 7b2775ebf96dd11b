// Split-KV flash-decode for head-heterogeneous attention on CUDA cores (Sec.
// 5, "Decode Stage", Eq. 8): one new token per sequence; retrieval KV heads
// attend over their whole history, streaming KV heads over their S sink + W
// window slots. This kernel serves d_head 64 (d_head 128 runs on the tensor
// cores, decode_tc.cu), including the d_head 64 H2Share reuse step, whose
// retrieval rows are borrowed positions gathered one row at a time.
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
#include "decode_common.cuh"
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
  static constexpr int NST = G <= 4 ? 6 : 5;    // pipeline stages
  static constexpr int STAGE_BYTES = TOK * RB * 2;
  static constexpr int DATA_BYTES = NST * STAGE_BYTES;
  static constexpr int OFF_MERGE = DATA_BYTES;   // [NW][G][D] o, [NW][G] m, [NW][G] l
  static constexpr int MERGE_BYTES = NW * G * (D + 2) * 4;
  static constexpr int OFF_BAR = (OFF_MERGE + MERGE_BYTES + 15) / 16 * 16;
  static constexpr int SMEM = OFF_BAR + 2 * NST * 8 + 32;
  static constexpr int THREADS = (NW + 1) * 32;
  static_assert(V % LPT == 0 && RP <= GP, "bad reduce-scatter shape");
  static_assert(THREADS * 8 <= DATA_BYTES, "scan scratch");
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
  float* mo = reinterpret_cast<float*>(smem + C::OFF_MERGE);  // [NW][G][D]
  float* mm = mo + C::NW * G * D;                              // [NW][G]
  float* ml = mm + C::NW * G;                                  // [NW][G]
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + NST;
  long long* sh64 = reinterpret_cast<long long*>(empty + NST);  // [0] total, [1] first offset
  int* sh32 = reinterpret_cast<int*>(sh64 + 2);                 // [0] first item, [1] combine flag
  volatile int* abort_flag = sh32 + 2;                          // set once any bounded wait gives up

  const CacheGeom& g = a.geom;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int HK = g.n_r + g.n_s;
  const int n_items = g.B * HK;
  const int P = a.n_ctas, p = blockIdx.x;

  // ---- every CTA finds its share of the concatenated rows and the first
  // item it touches (the ring memory is scratch here)
  dec::find_cta_range<C::THREADS>(a, reinterpret_cast<long long*>(smem), sh64, sh32);
  if (threadIdx.x == 0) {
#pragma unroll
    for (int s = 0; s < NST; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], C::NW);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const long long total = sh64[0];
  const long long start = (long long)p * total / P;
  const long long end = (long long)(p + 1) * total / P;
  const int first_id = sh32[0];
  const long long first_off = sh64[1];

  if (warp == C::NW) {
    // ------------------------------------------------------------ producer
    int it = 0;
    long long off = first_off;
    for (int id = first_id; id < n_items && off < end; ++id) {
      const int rows = dec::item_rows(a, id);
      const int lo = (int)(max(start, off) - off), hi = (int)(min(end, off + rows) - off);
      off += rows;
      if (lo >= hi) continue;
      const int b = id / HK, k = id - b * HK;
      const int kind = k < g.n_r ? 0 : 1, hi_idx = kind ? k - g.n_r : k;
      const int kvh = kind ? g.s_head[hi_idx] : g.r_head[hi_idx];
      const int t = __ldcg(&a.lens[b]);
      const int cap = kind ? g.S + g.W : g.max_seq;
      const int xr = kind == 0 ? t : (t < g.S ? t : g.S + (t - g.S) % g.W);
      const size_t reg = kind ? g.s_region(b, hi_idx) : g.r_region(b, hi_idx);
      const uint8_t* Kc = reinterpret_cast<const uint8_t*>(static_cast<const bf16*>(a.kv) + reg);
      const uint8_t* Vc = Kc + (size_t)cap * RB;
      const size_t new_off = ((size_t)b * g.Hkv + kvh) * D;
      const uint8_t* kn = reinterpret_cast<const uint8_t*>(static_cast<const bf16*>(a.k_new) + new_off);
      const uint8_t* vn = reinterpret_cast<const uint8_t*>(static_cast<const bf16*>(a.v_new) + new_off);
      // H2Share reuse step: the rows of a retrieval item are borrowed cache rows
      const bool indexed = a.idx != nullptr && kind == 0;
      const int32_t* rowlist =
          indexed ? a.idx + ((size_t)b * a.n_idx_groups + a.idx_map[hi_idx]) * a.top_k : nullptr;
      if ((indexed ? lo == 0 : (xr >= lo && xr < hi)) && lane < D / 8) {
        // append the new token (its row is read from the input below)
        reinterpret_cast<uint4*>(const_cast<uint8_t*>(Kc) + (size_t)xr * RB)[lane] =
            reinterpret_cast<const uint4*>(kn)[lane];
        reinterpret_cast<uint4*>(const_cast<uint8_t*>(Vc) + (size_t)xr * RB)[lane] =
            reinterpret_cast<const uint4*>(vn)[lane];
      }
      if (indexed) {
        // one 1D bulk copy per borrowed row, spread over the warp (lane l
        // copies rows l, l + 32, ... of a tile); indices are clamped to the
        // rows held, so a bad list cannot read out of bounds. A tile's
        // indices are loaded one tile ahead, while the producer waits for a
        // free stage: read at the tile itself, that load's latency under the
        // HBM stream would stall every stage.
        constexpr int RPL = TOK / 32;  // rows per lane and tile
        static_assert(TOK % 32 == 0, "tile rows");
        int nxt[RPL];
#pragma unroll
        for (int r = 0; r < RPL; ++r) nxt[r] = lo + r * 32 + lane < hi ? __ldg(rowlist + lo + r * 32 + lane) : 0;
        for (int row0 = lo; row0 < hi; row0 += TOK, ++it) {
          int cur[RPL];
#pragma unroll
          for (int r = 0; r < RPL; ++r) {
            cur[r] = nxt[r];
            const int j = row0 + TOK + r * 32 + lane;
            if (j < hi) nxt[r] = __ldg(rowlist + j);
          }
          const int st = it % NST;
          int ok = 1;
          if (lane == 0) {
            ok = !*abort_flag;
            if (ok && it >= NST && !mbar_wait(&empty[st], ((it / NST) & 1) ^ 1, a.err)) {
              *abort_flag = 1;
              ok = 0;
            }
          }
          if (!__shfl_sync(0xffffffffu, ok, 0)) break;
          const int cnt = min(TOK, hi - row0);
          if (lane == 0) mbar_arrive_expect_tx(&full[st], (uint32_t)cnt * RB * 2);
          __syncwarp();
          uint8_t* ks = smem + st * C::STAGE_BYTES;
#pragma unroll
          for (int r = 0; r < RPL; ++r) {
            const int rr = r * 32 + lane;
            if (rr < cnt) {
              const int cr = min(max(cur[r], 0), t);
              bulk_g2s(ks + (size_t)rr * RB, cr == xr ? kn : Kc + (size_t)cr * RB, RB, &full[st]);
              bulk_g2s(ks + (size_t)(TOK + rr) * RB, cr == xr ? vn : Vc + (size_t)cr * RB, RB, &full[st]);
            }
          }
          __syncwarp();
        }
      } else if (lane == 0) {
        for (int row0 = lo; row0 < hi && !*abort_flag; row0 += TOK, ++it) {
          const int st = it % NST;
          if (it >= NST && !mbar_wait(&empty[st], ((it / NST) & 1) ^ 1, a.err)) {
            *abort_flag = 1;
            break;
          }
          const int cnt = min(TOK, hi - row0);
          mbar_arrive_expect_tx(&full[st], (uint32_t)cnt * RB * 2);
          uint8_t* ks = smem + st * C::STAGE_BYTES;
          copy_rows<RB>(ks, Kc, kn, row0, cnt, xr, &full[st]);
          copy_rows<RB>(ks + TOK * RB, Vc, vn, row0, cnt, xr, &full[st]);
        }
      }
      __syncwarp();
      it = __shfl_sync(0xffffffffu, it, 0);  // lane 0 alone advanced it on a contiguous item
    }
    // every issued copy lands before the CTA can exit
    if (lane == 0)
      for (int j = it > NST ? it - NST : 0; j < it; ++j) mbar_wait(&full[j % NST], (j / NST) & 1, a.err);
  } else {
    // ------------------------------------------------------------ consumers
    const int gi = lane / C::LPT, c = lane % C::LPT;
    const int grp = warp * C::GPW + gi;
    const int tb = grp * C::NT;  // first tile row of this group
    int it = 0;
    long long off = first_off;
    for (int id = first_id; id < n_items && off < end; ++id) {
      const int rows = dec::item_rows(a, id);
      const long long item_off = off;
      const int lo = (int)(max(start, off) - off), hi = (int)(min(end, off + rows) - off);
      off += rows;
      if (lo >= hi) continue;
      const int b = id / HK, k = id - b * HK;
      const int kind = k < g.n_r ? 0 : 1;
      const int kvh = kind ? g.s_head[k - g.n_r] : g.r_head[k];

      float2 qf[G][4];
      float m[G], l[G];
      float2 o[G][4];
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

      for (int row0 = lo; row0 < hi; row0 += TOK, ++it) {
        const int st = it % NST;
        // warp-uniform: every lane leaves the loop together if a wait gave up
        bool stop = __any_sync(kFull, *abort_flag != 0);
        if (!stop) stop = !__all_sync(kFull, mbar_wait(&full[st], (it / NST) & 1, a.err));
        if (stop) {
          *abort_flag = 1;
          break;
        }
        const int cnt = min(TOK, hi - row0);
        const uint8_t* ks = smem + st * C::STAGE_BYTES;
        const uint8_t* vs = ks + TOK * RB;

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

        float s[C::RP], mx[C::RP];
#pragma unroll
        for (int kk = 0; kk < C::RP; ++kk) {
          const int v = c * C::RP + kk;
          const int tt = v / C::GP, r = v % C::GP;
          const bool valid = (tb + tt < cnt) && (r < G);
          s[kk] = valid ? part[kk] * a.scale_log2 : -INFINITY;
          mx[kk] = s[kk];
        }
#pragma unroll
        for (int msk = C::Q; msk < C::LPT; msk *= 2)
#pragma unroll
          for (int kk = 0; kk < C::RP; ++kk) mx[kk] = fmaxf(mx[kk], __shfl_xor_sync(kFull, mx[kk], msk));
        float bm[G];
#pragma unroll
        for (int j = 0; j < C::Q; ++j)
#pragma unroll
          for (int kk = 0; kk < C::RP; ++kk)
            if (j * C::RP + kk < G) bm[j * C::RP + kk] = __shfl_sync(kFull, mx[kk], gi * C::LPT + j);

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

        float pr[C::RP];
#pragma unroll
        for (int kk = 0; kk < C::RP; ++kk) {
          const int r = (c % C::Q) * C::RP + kk;
          float mr = m[0];
#pragma unroll
          for (int rr = 1; rr < G; ++rr) mr = (rr == r) ? m[rr] : mr;
          pr[kk] = (s[kk] == -INFINITY) ? 0.f : fast_exp2(s[kk] - mr);
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
            const float pv = __shfl_sync(kFull, pr[v % C::RP], gi * C::LPT + v / C::RP);
            l[r] += pv;
            const float2 pp = make_float2(pv, pv);
#pragma unroll
            for (int e = 0; e < 4; ++e) o[r][e] = __ffma2_rn(pp, vf[tt][e], o[r][e]);
          }
        }
      }

      // ---- merge the groups of each warp with shuffles, then the warps
#pragma unroll
      for (int msk = C::LPT; msk < 32; msk *= 2) {
#pragma unroll
        for (int r = 0; r < G; ++r) {
          const float m_o = __shfl_xor_sync(kFull, m[r], msk);
          const float l_o = __shfl_xor_sync(kFull, l[r], msk);
          const float M = fmaxf(m[r], m_o);
          const float wa = (m[r] == -INFINITY) ? 0.f : fast_exp2(m[r] - M);
          const float wb = (m_o == -INFINITY) ? 0.f : fast_exp2(m_o - M);
          l[r] = l[r] * wa + l_o * wb;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float ox = __shfl_xor_sync(kFull, o[r][e].x, msk);
            const float oy = __shfl_xor_sync(kFull, o[r][e].y, msk);
            o[r][e].x = o[r][e].x * wa + ox * wb;
            o[r][e].y = o[r][e].y * wa + oy * wb;
          }
          m[r] = M;
        }
      }
      if (gi == 0) {
#pragma unroll
        for (int r = 0; r < G; ++r) {
          float* dst = mo + ((size_t)warp * G + r) * D + c * 8;
#pragma unroll
          for (int e = 0; e < 4; ++e) *reinterpret_cast<float2*>(dst + 2 * e) = o[r][e];
          if (c == 0) {
            mm[warp * G + r] = m[r];
            ml[warp * G + r] = l[r];
          }
        }
      }
      named_barrier_sync(1, C::NW * 32);

      const int f = dec::cta_of(item_off, total, P), lst = dec::cta_of(item_off + rows - 1, total, P);
      const bool single = f == lst;
      const int slot = (p == f) ? 1 : 0;
      float* pbase = dec::partial_slot(a, p, slot, G, D);
      bf16* outp = static_cast<bf16*>(a.out) + ((size_t)b * g.Hq + (size_t)kvh * G) * D;
      for (int idx = threadIdx.x; idx < G * D; idx += C::NW * 32) {
        const int r = idx / D, d = idx - r * D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < C::NW; ++w) M = fmaxf(M, mm[w * G + r]);
        float O = 0.f, L = 0.f;
#pragma unroll
        for (int w = 0; w < C::NW; ++w) {
          const float mw = mm[w * G + r];
          const float wt = (mw == -INFINITY) ? 0.f : fast_exp2(mw - M);
          O += wt * mo[((size_t)w * G + r) * D + d];
          L += wt * ml[w * G + r];
        }
        if (single) {
          outp[idx] = __float2bfloat16_rn(O / L);
        } else {
          __stcg(pbase + idx, O);
          if (d == 0) {
            __stcg(pbase + G * D + r, M);
            __stcg(pbase + G * D + G + r, L);
          }
        }
      }
      if (!single) dec::merge_item<G, D, C::NW * 32, false>(a, p, f, lst, id, outp, mo, sh32 + 1);
      named_barrier_sync(1, C::NW * 32);
    }
  }

  // ---- the launch's last CTA advances the lengths
  __syncthreads();
  if (threadIdx.x == 0) dec::finish_launch(a, nullptr);
}

template <int D, int G>
cudaError_t launch_cfg(const DecodeArgs& a, cudaStream_t s) {
  using C = DecodeCfg<D, G>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  decode_kernel<C><<<a.n_ctas, C::THREADS, C::SMEM, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

bool decode_cc_supported(int D, int G) {
  return (D == 64 || D == 128) && (G == 1 || G == 2 || G == 4 || G == 7 || G == 8);
}

bool decode_supported(int D, int G) {
  if (D == 128) return decode_uses_tc(D, G);
  return decode_cc_supported(D, G);
}

// Two CTAs fit on an SM (about 100 KB of shared memory each), so 2 x SMs
// CTAs run as one wave; small launches use fewer, at least 256 rows each.
int decode_ctas(long long total_rows, int num_sms, int D, int G) {
  if (decode_uses_tc(D, G)) return decode_tc_ctas(total_rows, num_sms);
  return decode_cc_ctas(total_rows, num_sms);
}

int decode_cc_ctas(long long total_rows, int num_sms) {
  const long long by_rows = (total_rows + 255) / 256;
  long long p = 2LL * num_sms;
  if (by_rows < p) p = by_rows;
  return p < 1 ? 1 : (int)p;
}

size_t decode_partial_floats(int n_ctas, int G, int D) { return (size_t)n_ctas * 4 * dec::partial_stride(G, D); }

cudaError_t launch_decode_cc(const DecodeArgs& args, cudaStream_t s) {
  // this kernel walks its rows with unit weights and no item charge (its
  // loops count rows, not work units), so the split must use the same
  DecodeArgs a = args;
  a.gather_w = a.ring_w = 1;
  a.item_cost = 0;
  const int D = a.geom.D, G = a.geom.G;
  if (D == 128) {
    switch (G) {
      case 1: return launch_cfg<128, 1>(a, s);
      case 2: return launch_cfg<128, 2>(a, s);
      case 4: return launch_cfg<128, 4>(a, s);
      case 7: return launch_cfg<128, 7>(a, s);
      case 8: return launch_cfg<128, 8>(a, s);
    }
  } else if (D == 64) {
    switch (G) {
      case 1: return launch_cfg<64, 1>(a, s);
      case 2: return launch_cfg<64, 2>(a, s);
      case 4: return launch_cfg<64, 4>(a, s);
      case 7: return launch_cfg<64, 7>(a, s);
      case 8: return launch_cfg<64, 8>(a, s);
    }
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t s) {
  if (decode_uses_tc(a.geom.D, a.geom.G)) return launch_decode_tc(a, s);
  return launch_decode_cc(a, s);
}

}  // namespace aoh
