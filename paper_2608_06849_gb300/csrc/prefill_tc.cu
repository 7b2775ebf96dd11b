// Causal prefill attention on tcgen05 tensor cores (Sec. 5, "Chunked-Prefill
// Stage", with the per-token sink + window rule for streaming heads). A call
// processes one chunk of every sequence: rows at positions Lb .. Lb + len - 1
// after Lb cached tokens (Lb = 0 for a first prefill). Cached keys are read
// from the KV cache itself (retrieval rows, or the streaming sink + ring
// slots) before the chunk's own keys; the cache is appended after this
// kernel, so the ring still holds the positions the chunk's rows need.
//
// One CTA computes two consecutive 128-row query tiles (A = rows q0..q0+127,
// B = rows q0+128..q0+255) of one query head against the same stream of
// 128-key K/V tiles. The KV tiles visited come from a per-head schedule: a
// retrieval head visits tiles 0 .. causal end; a streaming head only the
// tiles holding its S sinks and the tiles that intersect the W-token window
// of some row, so its cost is O(S + W) per row instead of O(T). Both query
// tiles visit the union of their tile sets; a tile hidden from every row of
// one query tile contributes zero weights there. Tiles fully visible to every
// row of a query tile skip the mask.
//
// Warp roles (320 threads):
//   warp 0      TMA producer: Q_A, Q_B once, then K_j / V_j tiles into a
//               4-stage ring (4D tensor maps over [B][T][H][D], 128-byte swizzle).
//   warp 1      TMEM owner and MMA issuer. S_X(j) = Q_X K_j^T reads both
//               operands from shared memory; O_X += P_X(j) V_j reads P_X from
//               TMEM, where the softmax wrote it over the first 64 columns of
//               S_X. Per KV tile the issue order is O_A += P_A V, S_A(j+1),
//               O_B += P_B V, S_B(j+1): a tile's next S overwrites its P only
//               after the P.V that reads it (MMAs of one thread run in order),
//               and while one query tile's softmax runs the tensor pipe works
//               on the other's MMAs, hiding the commit -> softmax -> issue
//               latency of each tile.
//   warps 2-5   softmax of tile A, warps 6-9 softmax of tile B: thread r owns
//               row r (TMEM lane r). One tcgen05.ld pass reads its S row, a
//               two-range integer mask hides keys, max and sum reduce in 8
//               independent chains, p = 2^(s*scale - m) costs one FFMA and one
//               EX2, the running max moves only when it grows by more than
//               2^8 (O rarely rescaled), and bf16 P pairs go back to TMEM with
//               tcgen05.st (key k in column k/2, even k in the low half).
// TMEM columns: S_A / P_A [0,128), S_B / P_B [128,256), O_A [256, 256+D),
// O_B [256+D, 256+2D).
#include <math.h>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace aoh {
namespace {

using bf16 = __nv_bfloat16;
constexpr int kBM = 128;         // rows per query tile (a CTA owns two)
constexpr int kBN = 128;         // keys per KV tile
constexpr int kNS = 4;           // KV ring stages (K and V tiles alternate)
constexpr float kRescaleThreshold = 8.0f;
constexpr uint32_t kTmemCols = 512;
constexpr int kThreads = 320;

template <int D>
struct PfCfg {
  static constexpr int DBLK = D / 64;            // 64-wide column blocks (one TMA box each)
  static constexpr int BOX = 128 * 64 * 2;       // bytes of one [128 rows][64] box
  static constexpr int QBYTES = DBLK * BOX;      // one query tile
  static constexpr int KVBYTES = DBLK * BOX;
  static constexpr int OFF_Q = 0;                // Q_A, Q_B
  static constexpr int OFF_KV = OFF_Q + 2 * QBYTES;
  static constexpr int OFF_BAR = OFF_KV + kNS * KVBYTES;
  static constexpr int NBAR = 1 + 2 * kNS + 2 + 2 + 2 + 2 + 1 + 2;
  static constexpr int SMEM = OFF_BAR + NBAR * 8 + 16 + 1024;
  static constexpr uint32_t IDESC_S = idesc_bf16(kBM, kBN, false);
  static constexpr uint32_t IDESC_PV = idesc_bf16(kBM, D, true);
  static_assert(SMEM <= 232448, "shared memory");
  static_assert(256 + 2 * D <= (int)kTmemCols, "TMEM columns");
};

// Bits lo..hi-1 of a 32-bit word (lo, hi clamped to [0, 32]).
__device__ __forceinline__ uint32_t range_bits(int lo, int hi) {
  lo = max(lo, 0);
  hi = min(hi, 32);
  if (hi <= lo) return 0u;
  const uint32_t top = hi == 32 ? 0xffffffffu : ((1u << hi) - 1u);
  return top & ~((1u << lo) - 1u);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) prefill_tc_kernel(const __grid_constant__ PrefillTcArgs a) {
  using C = PfCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sKV = smem + C::OFF_KV;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;
  uint64_t* kv_empty = kv_full + kNS;
  uint64_t* s_full = kv_empty + kNS;  // [2]: S_A, S_B ready
  uint64_t* s_empty = s_full + 2;     // [2]: S_A, S_B read by the softmax
  uint64_t* p_full = s_empty + 2;     // [2]: P_A, P_B written
  uint64_t* pv_done = p_full + 2;     // [2]: O_A, O_B updated (P buffer free)
  uint64_t* drain = pv_done + 2;
  // [2]: padding rows of the item's first / second partial V tile are zeroed.
  // Only the last cache tile and the chunk tile holding row len - 1 can be
  // partial, so each barrier completes at most once per item.
  uint64_t* v_zeroed = drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(v_zeroed + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int4 item = a.work[blockIdx.x];
  const int b = item.x, h = item.y, q0 = item.z;
  const CacheGeom& g = a.geom;
  const int kvh = h / g.G;
  const bool streaming = g.kind[kvh] != 0;
  const int len = a.lens[b];
  const int Lb = a.base[b];
  const int q_end = min(q0 + 2 * kBM, len);
  const int S_rel = g.S - Lb;
  const int n_c = Lb == 0 ? 0 : ((streaming ? min(Lb, g.S + g.W) : Lb) + kBN - 1) / kBN;
  // KV tiles visited (union of both query tiles): [0, a_end) then [c_begin, c_end)
  int a_end, c_begin, c_end;
  if (!streaming) {
    a_end = (q_end + kBN - 1) / kBN;
    c_begin = c_end = a_end;
  } else {
    a_end = (min(max(S_rel, 0), q_end) + kBN - 1) / kBN;
    c_begin = max(a_end, max(0, g.wstart(q0)) / kBN);
    c_end = max(c_begin, (q_end + kBN - 1) / kBN);
  }
  const int n_tiles = n_c + a_end + (c_end - c_begin);
  // keys of KV tile jj that hold data (the rest: cache rows not yet written,
  // or chunk padding); fewer than kBN makes the tile partial
  auto tile_valid = [&](int jj) {
    if (jj < n_c) return (streaming ? min(Lb, g.S + g.W) : Lb) - jj * kBN;
    const int jc = jj - n_c;
    return len - (jc < a_end ? jc : c_begin + (jc - a_end)) * kBN;
  };

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < kNS; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(&s_full[x], 1);
      mbar_init(&s_empty[x], 4);
      mbar_init(&p_full[x], 4);
      mbar_init(&pv_done[x], 1);
    }
    mbar_init(drain, 1);
    mbar_init(&v_zeroed[0], 1);
    mbar_init(&v_zeroed[1], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // Lane 0 issues the copies. Rows of a V tile past its valid keys may hold
    // anything (cache rows not yet written, chunk padding) and a zero weight
    // times a NaN is still NaN, so for a partial V tile the whole warp waits
    // for the copy, zeroes those rows and signals v_zeroed before the MMA
    // issuer may read the tile.
    if (lane == 0) {
      prefetch_tmap(&a.tq);
      prefetch_tmap(&a.tk);
      prefetch_tmap(&a.tv);
      mbar_arrive_expect_tx(q_full, 2 * C::QBYTES);
      for (int x = 0; x < 2; ++x)
        for (int db = 0; db < C::DBLK; ++db)
          tma_load_4d(sQ + x * C::QBYTES + db * C::BOX, &a.tq, db * 64, h, q0 + x * kBM, b, q_full);
    }
    int issued = 0, n_partial = 0;
    bool ok = true;
    for (int jj = 0; jj < n_tiles && ok; ++jj) {
      const int jc = jj - n_c;
      const int j = jc < a_end ? jc : c_begin + (jc - a_end);
      for (int sel = 0; sel < 2; ++sel) {
        const int it = 2 * jj + sel;
        const int st = it % kNS;
        if (lane == 0) {
          if (it >= kNS && !wait_bar(&kv_empty[st], ((it / kNS) & 1) ^ 1, a.err, abort_flag)) {
            ok = false;
          } else {
            mbar_arrive_expect_tx(&kv_full[st], C::KVBYTES);
            if (jj < n_c) {
              // cache region viewed as [regions][K, V][rows][D]
              const CUtensorMap* map = streaming ? &a.tcs : &a.tcr;
              const int region = streaming ? b * g.n_s + g.idx[kvh] : b * g.n_r + g.idx[kvh];
              for (int db = 0; db < C::DBLK; ++db)
                tma_load_4d(sKV + st * C::KVBYTES + db * C::BOX, map, db * 64, jj * kBN, sel, region,
                            &kv_full[st]);
            } else {
              const CUtensorMap* map = sel ? &a.tv : &a.tk;
              for (int db = 0; db < C::DBLK; ++db)
                tma_load_4d(sKV + st * C::KVBYTES + db * C::BOX, map, db * 64, kvh, j * kBN, b, &kv_full[st]);
            }
            issued = it + 1;
          }
        }
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        const int valid = tile_valid(jj);
        if (sel == 1 && valid < kBN && n_partial < 2) {
          if (!__all_sync(0xffffffffu, wait_bar(&kv_full[st], (it / kNS) & 1, a.err, abort_flag))) {
            ok = false;
            break;
          }
          uint8_t* vt = sKV + st * C::KVBYTES;
          for (int idx = max(valid, 0) * 8 + lane; idx < kBN * 8; idx += 32) {  // 16-byte chunks
            const int row = idx >> 3, chunk = idx & 7;
#pragma unroll
            for (int db = 0; db < C::DBLK; ++db)
              *reinterpret_cast<uint4*>(vt + db * C::BOX + row * 128 + chunk * 16) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&v_zeroed[n_partial]);
          ++n_partial;
        }
      }
    }
    // every issued copy lands before the CTA can exit
    if (lane == 0) {
      drain_wait(q_full, 0, a.err);
      for (int it = issued > kNS ? issued - kNS : 0; it < issued; ++it)
        drain_wait(&kv_full[it % kNS], (it / kNS) & 1, a.err);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t q_addr = smem_u32(sQ), kv_addr = smem_u32(sKV);
      auto issue_s = [&](int x, int jj) {
        const uint32_t k_addr = kv_addr + ((2 * jj) % kNS) * C::KVBYTES;
        const uint32_t qa = q_addr + x * C::QBYTES;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(qa + (kk >> 2) * C::BOX + (kk & 3) * 32, 16, 1024);
          const uint64_t bd = sdesc_sw128(k_addr + (kk >> 2) * C::BOX + (kk & 3) * 32, 16, 1024);
          tc_mma(tmem + x * 128, ad, bd, C::IDESC_S, kk > 0 ? 1u : 0u);
        }
        tc_commit(&s_full[x]);
      };
      auto issue_pv = [&](int x, int jj) {
        const uint32_t v_addr = kv_addr + ((2 * jj + 1) % kNS) * C::KVBYTES;
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          const uint64_t bd = sdesc_sw128(v_addr + kk * 16 * 128, C::BOX, 1024);
          tc_mma_ts(tmem + 256 + x * D, tmem + x * 128 + kk * 8, bd, C::IDESC_PV, (jj > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&pv_done[x]);
      };
      auto wait_k = [&](int jj) { return wait_bar(&kv_full[(2 * jj) % kNS], ((2 * jj) / kNS) & 1, a.err, abort_flag); };
      int n_partial = 0;  // partial V tiles seen so far (index into v_zeroed)
      auto wait_v = [&](int jj) {
        if (!wait_bar(&kv_full[(2 * jj + 1) % kNS], ((2 * jj + 1) / kNS) & 1, a.err, abort_flag)) return false;
        if (tile_valid(jj) < kBN && n_partial < 2) {
          if (!wait_bar(&v_zeroed[n_partial], 0, a.err, abort_flag)) return false;
          ++n_partial;
        }
        return true;
      };
      bool ok = wait_bar(q_full, 0, a.err, abort_flag) && wait_k(0);
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        issue_s(1, 0);
        tc_commit(&kv_empty[0]);
      }
      for (int jj = 0; jj < n_tiles && ok; ++jj) {
        const bool more = jj + 1 < n_tiles;
        const uint32_t ph = jj & 1;
        // tile A: P_A(jj) sits in S_A's columns; S_A(jj+1) may overwrite them
        // only after O_A += P_A(jj) V_jj is issued (same-thread MMAs run in order)
        if (!wait_v(jj) || !wait_bar(&p_full[0], ph, a.err, abort_flag)) { ok = false; break; }
        tc_fence_after();
        issue_pv(0, jj);
        if (more) {
          if (!wait_k(jj + 1)) { ok = false; break; }
          tc_fence_after();
          issue_s(0, jj + 1);
        }
        if (!wait_bar(&p_full[1], ph, a.err, abort_flag)) { ok = false; break; }
        tc_fence_after();
        issue_pv(1, jj);
        tc_commit(&kv_empty[(2 * jj + 1) % kNS]);
        if (more) {
          issue_s(1, jj + 1);
          tc_commit(&kv_empty[(2 * (jj + 1)) % kNS]);
        }
      }
      tc_commit(drain);
      drain_wait(drain, 0, a.err);
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int x = (warp - 2) >> 2;        // 0: tile A (warps 2-5), 1: tile B (warps 6-9)
    const int q4 = warp & 3;              // TMEM lane quarter this warp may access
    const int r = q4 * 32 + lane;
    const int qx0 = q0 + x * kBM;         // first row of this query tile
    const int i = qx0 + r;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t s_col = x * 128, o_col = 256 + x * D;
    const int S = g.S, W = g.W;
    const int rot = (streaming && Lb > S + W) ? (Lb - S) % W : 0;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int jj = 0; jj < n_tiles; ++jj) {
      const int jc = jj - n_c;
      const int j = jj < n_c ? jj : (jc < a_end ? jc : c_begin + (jc - a_end));
      const int j0 = j * kBN;
      if (!__all_sync(0xffffffffu, wait_bar(&s_full[x], jj & 1, a.err, abort_flag))) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[kBN];
      {
        uint32_t v0[32], v1[32], v2[32], v3[32];
        tmem_ld32(tl + s_col, v0);
        tmem_ld32(tl + s_col + 32, v1);
        tmem_ld32(tl + s_col + 64, v2);
        tmem_ld32(tl + s_col + 96, v3);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          s[e] = __uint_as_float(v0[e]);
          s[32 + e] = __uint_as_float(v1[e]);
          s[64 + e] = __uint_as_float(v2[e]);
          s[96 + e] = __uint_as_float(v3[e]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[x]);

      // hidden keys -> -inf. In tile coordinates key k is visible iff
      // k <= kmax (causal and inside the sequence) and, for a streaming head,
      // k < ks (a sink) or k >= kw (inside the window).
      // Hidden keys -> -inf. Every tile kind reduces to visible key ranges
      // [e_lo, e_hi), [a0, a1), [b0, b1) in tile coordinates, turned into four
      // 32-bit masks (one per 32 keys) so that each score costs one AND with
      // an immediate and one select.
      bool need_mask;
      int e_hi = kBN, a0 = 0, a1 = 0, b0 = 0, b1 = 0;
      if (jj < n_c) {
        if (!streaming) {
          need_mask = j0 + kBN > Lb;
          e_hi = Lb - j0;
        } else {
          need_mask = true;
          e_hi = min(S, Lb) - j0;
          // cached positions the row may see: sinks, and [Lb + wstart(i), Lb)
          const int skip = W + g.wstart(i);  // oldest ring positions hidden
          if (Lb <= S + W) {
            a0 = max(S, Lb + g.wstart(i)) - j0;
            a1 = Lb - j0;
          } else if (skip < W) {
            const int u = rot + max(skip, 0);
            if (u < W) {
              a0 = S + u - j0;
              a1 = S + W - j0;
              b0 = S - j0;
              b1 = S + rot - j0;
            } else {
              a0 = S + u - W - j0;
              a1 = S + rot - j0;
            }
          }
        }
      } else {
        const int jl = j0 + kBN - 1;
        need_mask = !(jl <= qx0 && jl < len && (!streaming || jl < S_rel || j0 >= g.wstart(qx0 + kBM - 1)));
        const int kmax = min(i, len - 1) - j0;
        if (!streaming) {
          e_hi = kmax + 1;
        } else {
          e_hi = min(kmax + 1, S_rel - j0);
          a0 = g.wstart(i) - j0;
          a1 = kmax + 1;
        }
      }
      if (need_mask) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const uint32_t vm = range_bits(0, e_hi - 32 * c) | range_bits(a0 - 32 * c, a1 - 32 * c) |
                              range_bits(b0 - 32 * c, b1 - 32 * c);
#pragma unroll
          for (int e = 0; e < 32; ++e) s[32 * c + e] = (vm & (1u << e)) ? s[32 * c + e] : -INFINITY;
        }
      }
      // row max of the raw scores (the scale is positive): 8 chains of
      // three-input max
      float mx8[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mx8[u] = fmaxf(s[u], s[u + 8]);
#pragma unroll
      for (int k = 16; k < kBN; k += 16)
#pragma unroll
        for (int u = 0; u < 8; ++u) mx8[u] = fmax3f(mx8[u], s[k + u], s[k + 8 + u]);
      const float rmax = fmax3f(fmax3f(mx8[0], mx8[1], mx8[2]), fmax3f(mx8[3], mx8[4], mx8[5]),
                                fmaxf(mx8[6], mx8[7])) *
                         a.scale_log2;
      const float mn = fmaxf(m, rmax);
      const bool resc = mn > m + kRescaleThreshold;
      float alpha = 1.f;
      if (resc) {
        alpha = (m == -INFINITY) ? 0.f : fast_exp2(m - mn);
        m = mn;
      }
      const bool warp_resc = __any_sync(0xffffffffu, resc) && jj > 0;
      const float neg_m = (m == -INFINITY) ? 0.f : -m;

      // p = 2^(s * scale - m), hidden keys give 0. Packed f32x2 arithmetic: one
      // FFMA2 forms two exponent arguments and one FADD2 adds two weights into
      // one of four pair accumulators. bf16 pairs (key k in column k/2, even k
      // low) are written over the first 64 columns of this tile's S in TMEM.
      const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
      const float2 nm2 = make_float2(neg_m, neg_m);
      float2 sum4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) sum4[u] = make_float2(0.f, 0.f);
#pragma unroll
      for (int hh = 0; hh < 4; ++hh) {
        uint32_t w[16];
#pragma unroll
        for (int t = 0; t < 16; ++t) {
          const int k = hh * 32 + 2 * t;
          const float2 e = __ffma2_rn(make_float2(s[k], s[k + 1]), sc2, nm2);
          const float2 pp = make_float2(fast_exp2(e.x), fast_exp2(e.y));
          sum4[t & 3] = __fadd2_rn(sum4[t & 3], pp);
          w[t] = float2_to_bf16x2(pp.x, pp.y);
        }
        tmem_st16(tl + s_col + hh * 16, w);
      }
      const float2 s01 = __fadd2_rn(sum4[0], sum4[1]), s23 = __fadd2_rn(sum4[2], sum4[3]);
      const float2 s03 = __fadd2_rn(s01, s23);
      const float sum = s03.x + s03.y;
      l = l * alpha + sum;

      // rescale O (rare): O_X += P_X(jj-1) V must have landed first
      if (warp_resc) {
        if (!__all_sync(0xffffffffu, wait_bar(&pv_done[x], (jj - 1) & 1, a.err, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(tl + o_col + c * 32, v);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * alpha);
          tmem_st32(tl + o_col + c * 32, v);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[x]);
    }
    if (ok && __all_sync(0xffffffffu, wait_bar(&pv_done[x], (n_tiles - 1) & 1, a.err, abort_flag))) {
      tc_fence_after();
      const float inv = 1.f / l;
      bf16* op = static_cast<bf16*>(a.out) + (((size_t)b * a.T + min(i, len - 1)) * g.Hq + h) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(tl + o_col + c * 32, v);
        tmem_ld_wait();
        if (i < len) {
#pragma unroll
          for (int e = 0; e < 32; e += 8) {
            uint4 w;
            w.x = float2_to_bf16x2(__uint_as_float(v[e + 0]) * inv, __uint_as_float(v[e + 1]) * inv);
            w.y = float2_to_bf16x2(__uint_as_float(v[e + 2]) * inv, __uint_as_float(v[e + 3]) * inv);
            w.z = float2_to_bf16x2(__uint_as_float(v[e + 4]) * inv, __uint_as_float(v[e + 5]) * inv);
            w.w = float2_to_bf16x2(__uint_as_float(v[e + 6]) * inv, __uint_as_float(v[e + 7]) * inv);
            *reinterpret_cast<uint4*>(op + c * 32 + e) = w;
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

namespace {

// 4D map over a [B][T][H][D] bf16 tensor, box [1][128][1][64], 128-byte swizzle.
bool make_map(CUtensorMap* map, const void* base, int B, int T, int H, int D) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)T, (cuuint64_t)B};
  cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2, (cuuint64_t)T * H * D * 2};
  cuuint32_t box[4] = {64, 1, 128, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int D>
cudaError_t launch_cfg(const PrefillTcArgs& a, int n_items, cudaStream_t s) {
  using C = PfCfg<D>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(prefill_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  prefill_tc_kernel<D><<<n_items, kThreads, C::SMEM, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

bool prefill_tc_make_maps(PrefillTcArgs* a, const void* q, const void* k, const void* v, int B, int T) {
  const CacheGeom& g = a->geom;
  return make_map(&a->tq, q, B, T, g.Hq, g.D) && make_map(&a->tk, k, B, T, g.Hkv, g.D) &&
         make_map(&a->tv, v, B, T, g.Hkv, g.D);
}

// 4D map over one kind of cache region: [regions][K, V][cap rows][D], box
// [1][1][128][64], 128-byte swizzle. Rows past `cap` read as zeros.
static bool make_region_map(CUtensorMap* map, const void* base, int regions, int cap, int D) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)cap, 2, (cuuint64_t)regions};
  cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)cap * D * 2, (cuuint64_t)cap * D * 2 * 2};
  cuuint32_t box[4] = {64, 128, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_cache_region_maps(CUtensorMap* tcr, CUtensorMap* tcs, const CacheGeom& g, const void* kv) {
  const bf16* base = static_cast<const bf16*>(kv);
  bool ok = true;
  if (g.n_r > 0) ok = ok && make_region_map(tcr, base + g.r_region(0, 0), g.B * g.n_r, g.max_seq, g.D);
  if (g.n_s > 0) ok = ok && make_region_map(tcs, base + g.s_region(0, 0), g.B * g.n_s, g.S + g.W, g.D);
  return ok;
}

bool prefill_tc_make_cache_maps(PrefillTcArgs* a, const void* kv) {
  return make_cache_region_maps(&a->tcr, &a->tcs, a->geom, kv);
}

cudaError_t launch_prefill_tc(const PrefillTcArgs& a, int n_items, cudaStream_t s) {
  if (n_items <= 0) return cudaSuccess;
  if (a.geom.D == 128) return launch_cfg<128>(a, n_items, s);
  if (a.geom.D == 64) return launch_cfg<64>(a, n_items, s);
  return cudaErrorInvalidValue;
}

}  // namespace aoh
