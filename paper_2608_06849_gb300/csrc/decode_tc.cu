// Split-KV decode on tcgen05 tensor cores (Sec. 5, "Decode Stage", Eq. 8;
// d_head = 128, GQA groups of 1-8 and 16). With G query heads per KV head,
// every cached K/V row meets G queries: 4*G*d flops per 4*d bytes. On CUDA
// cores that arithmetic (plus the shuffles that reduce the dot products)
// stops hiding under the HBM stream above g = 4, and even at g = 4 it costs a
// few percent; here it runs as two skinny MMAs per 128-key tile, with the G
// heads padded to N = 16:
//
//   S^T[128 keys][16]  = K_tile[128][d] . Q^T           (A = K, K-major; B = Q, K-major)
//   O^T[d][16]        += V_tile^T[d][128] . P^T[128][16] (A = V, MN-major; B = P, K-major)
//
// Both accumulators live in TMEM: S^T in one of two 16-column buffers (row =
// key), O^T in 16 more columns (row = d). The split of the step's rows over
// CTAs, the partial format and the merge are those of the CUDA-core kernel
// (decode_common.cuh); one CTA per SM.
//
// Warp roles (192 threads; 704 in the reuse step's variant for G <= 4, 448
// above):
//   warps 0-3  softmax: thread t owns key t of the tile (TMEM lane t). It
//              reads its 16 scores, hides keys past the tile's valid rows,
//              takes the per-head tile maximum (warp redux, then the four
//              warps through shared memory), moves the running maximum only
//              when it grows by more than 2^8 (then rescales its row d = t of
//              O^T in TMEM), forms p = 2^(s - m) and writes P^T as bf16 into a
//              swizzled K-major [16][128] buffer. Per-thread partial sums of p
//              are reduced once per item. Rows past the valid keys of a tail V
//              tile are zeroed first: they may hold unwritten cache rows and a
//              zero weight times a NaN is NaN.
//   warp 4     TMA producer: K and V tiles of one (sequence, KV head) region
//              into a 3-stage ring (4D tensor maps over the cache regions,
//              128-byte swizzle, rows past the region read as zeros).
//   warps 6-21 (6-13 for G > 4; the H2Share reuse step's variant) gather
//              warps: a retrieval item's rows are borrowed positions, which
//              these warps copy with 16-byte cp.async copies into the same
//              swizzled ring, 8 (16) rows of each tile per warp; the CTAs
//              split the step's rows with each gathered row weighing 3/2
//              contiguous rows (a row gather costs more than its share of a
//              streamed tile). The MMA warp issues a gathered tile's P V
//              right after its P, which frees the ring stage for the next
//              gather one tile earlier.
//   warp 5     TMEM owner and MMA issuer. Loads each item's Q into one of two
//              swizzled buffers, writes the new token's K/V row over its
//              (stale) cache row in the landed tile and appends it to the
//              cache, issues S(j) and then O += P(j-1) V(j-1).
#include <math.h>

#include "common.cuh"
#include "decode_common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace aoh {
namespace {

using bf16 = __nv_bfloat16;
constexpr int kD = 128;
constexpr int kBN = 128;                   // keys per tile
constexpr int kN = 16;                     // N of both MMAs (query heads, padded)
constexpr int kNS = 3;                     // ring stages
constexpr int kThreads = 192;              // warps 0-5 (see the file comment)
constexpr int kSoftmaxThreads = 128;
constexpr uint32_t kTmemCols = 64;         // S[0] [0,16), S[1] [16,32), O [32,48)
constexpr uint32_t kOcol = 32;
constexpr float kRescaleThreshold = 8.0f;  // log2 units
// Rows charged for a switch from one item to the next (DecodeArgs::
// item_cost), in steps whose CTAs hold fewer than kItemCostMaxShare rows
// each. A CTA that switches finishes its first item's epilogue and arrival
// before the next item's softmax can go on, so with an equal share it ends
// last, and then also runs the second item's merge. Measured with B=1,
// Qwen2.5-7B shape (2 of 4 KV heads streaming), us per step, mean over six
// lengths T .. T + 331 (cost 0 / 256 / 384 / 512 / 768 rows): 4K 16.9 /
// 16.9 / 16.2 / 15.4 / 14.9, 8K 23.2 / 20.5 / 17.8 / 17.0 / 15.7, 16K 19.9
// / 17.8 / 17.3 / 17.3 / 17.4, 32K 21.7 / 18.1 / 18.0 / 17.8 / 17.8, 64K
// 24.7 / 23.8 / 22.7 / 22.9 / 22.9, 128K 38.2 / - / 36.9 / 37.5 / 37.5;
// through the 28-layer stack per token (CUDA graph; cost 384 / 512 / 768):
// 4K 439 / 432 / 399, 32K 531 / 531 / 528, 128K 973 / 1037 / 1030.
// Steps on fewer CTAs than SMs (4K, 8K: at least 512 rows per CTA, few
// items) gain from the larger charge, which moves item starts onto CTA
// boundaries; steps on every SM keep 384. Llama-3-8B shape at B=16, 128K
// (29K rows per CTA): 628 us with no charge, 629-630 with 256 rows.
constexpr int kItemCost = 384;
constexpr int kItemCostFewCtas = 768;
constexpr long long kItemCostMaxShare = 16384;
constexpr int kBox = kBN * 64 * 2;         // one [128 rows][64] TMA box, 16 KB
constexpr int kTile = 2 * kBox;            // a K or V tile (d = 128)
constexpr int kStage = 2 * kTile;          // K then V
constexpr int kOpBuf = 2 * kN * 128;       // [16 rows][128] bf16 operand, two 64-wide blocks
constexpr int OFF_KV = 0;
constexpr int OFF_Q = OFF_KV + kNS * kStage;
constexpr int OFF_P = OFF_Q + 2 * kOpBuf;
constexpr int OFF_RED = OFF_P + 2 * kOpBuf;   // [2][4][16] warp maxima, [4][16] warp sums
constexpr int OFF_MS = OFF_RED + (2 * 64 + 64) * 4;
constexpr int MS_FLOATS = 1024;               // merge scratch
constexpr int OFF_BAR = OFF_MS + MS_FLOATS * 4;
constexpr int NBAR = 3 * kNS + 2 + 2 + 2 + 2 + 1 + 1;
constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
constexpr int kLensCap = 2048;                // sequence lengths mirrored in shared memory
constexpr int OFF_LENS = OFF_MISC + 64;
constexpr int SMEM = OFF_LENS + kLensCap * 4 + 1024;
constexpr uint32_t IDESC_S = idesc_bf16(kBN, kN, false, false);
constexpr uint32_t IDESC_PV = idesc_bf16(kD, kN, false, true);
static_assert(SMEM <= 232448, "shared memory");
static_assert(OFF_Q % 1024 == 0 && OFF_P % 1024 == 0, "operand alignment");

// Gather warps of the H2Share reuse variant (warps 6 on). The cp.async
// copies a warp keeps in flight are bounded per warp, so the gather rate
// grows with the warps that issue them: sixteen for groups of up to four
// heads (704 threads, 80 registers each), eight above, where the wider
// group's softmax state needs more registers per thread.
__host__ __device__ constexpr int gather_warps(int G, bool gather) { return gather ? (G <= 4 ? 16 : 8) : 0; }
static_assert((kThreads + 32 * 16) * 8 <= kNS * kStage, "scan scratch");

// GATHER: the H2Share reuse variant, whose gather warps copy the borrowed
// rows of retrieval items (a.idx != nullptr); the producer warp then loads
// only the contiguous (streaming) tiles.
template <int G, bool GATHER>
__global__ void __launch_bounds__(kThreads + 32 * gather_warps(G, GATHER), 1)
    decode_tc_kernel(const __grid_constant__ DecodeArgs a) {
  static_assert(G >= 1 && G <= kN, "group size");
  constexpr int GW = gather_warps(G, GATHER);
  constexpr int RPW = GATHER ? kBN / GW : kBN;  // rows of each tile a gather warp copies
  constexpr int NT = kThreads + 32 * GW;
  static_assert(2 * (dec::kGroup + 8) * G + 2 * G <= MS_FLOATS, "merge scratch");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
  uint8_t* sKV = smem + OFF_KV;
  uint8_t* sQ = smem + OFF_Q;
  uint8_t* sP = smem + OFF_P;
  float* red = reinterpret_cast<float*>(smem + OFF_RED);  // [2][4][16]
  float* lsum = red + 2 * 64;                             // [4][16]
  float* ms = reinterpret_cast<float*>(smem + OFF_MS);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + OFF_BAR);  // [kNS] a TMA-loaded tile landed
  uint64_t* empty = full + kNS;
  uint64_t* gfull = empty + kNS;    // [kNS] a gathered tile landed (reuse variant)
  uint64_t* s_full = gfull + kNS;   // [2] S(j) in TMEM
  uint64_t* s_free = s_full + 2;    // [2] S(j) read by the softmax
  uint64_t* p_full = s_free + 2;    // [2] P(j) written
  uint64_t* p_free = p_full + 2;    // [2] O += P(j) V(j) done
  uint64_t* o_free = p_free + 2;    // the item's final O read
  uint64_t* drain = o_free + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  long long* sh64 = reinterpret_cast<long long*>(smem + OFF_MISC + 8);  // [0] total, [1] first offset
  int* sh32 = reinterpret_cast<int*>(sh64 + 2);                         // [0] first item, [1] merge flag
  int* lens_s = reinterpret_cast<int*>(smem + OFF_LENS);

  const CacheGeom& g = a.geom;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int HK = g.n_r + g.n_s;
  const int n_items = g.B * HK;
  const int P = a.n_ctas, p = blockIdx.x;

  // Prologue that touches no global memory; it may overlap the tail of the
  // previous kernel on the stream (programmatic dependent launch).
  // Q and P rows >= G stay zero for the whole launch
  for (int i = threadIdx.x; i < 4 * kOpBuf / 16; i += NT)
    reinterpret_cast<uint4*>(sQ)[i] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  if (threadIdx.x == 0) {
    for (int s = 0; s < kNS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&gfull[s], GATHER ? GW : 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(&s_full[x], 1);
      mbar_init(&s_free[x], 4);
      mbar_init(&p_full[x], 4);
      mbar_init(&p_free[x], 1);
    }
    mbar_init(o_free, 4);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 5) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // everything the previous kernels wrote (lengths, cache, inputs, counters)
  // is visible after this wait; the next step may then start its prologue
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // the lengths cannot change during the launch (the last CTA to finish
  // advances them), so every role reads this copy
  const int* ls = g.B <= kLensCap ? lens_s : nullptr;
  if (ls != nullptr) {
    for (int i = threadIdx.x; i < g.B; i += NT) lens_s[i] = __ldcg(&a.lens[i]);
    __syncthreads();
  }
  dec::find_cta_range<NT>(a, reinterpret_cast<long long*>(sKV), sh64, sh32, ls);
  __syncthreads();
  const long long total = sh64[0];
  const long long start = (long long)p * total / P;
  const long long end = (long long)(p + 1) * total / P;
  const int first_id = sh32[0];
  const long long first_off = sh64[1];

  if (warp == 4) {
    // ------------------------------------------------------------ producer
    // Lane 0 loads 128-row K and V tiles of the region (4D tensor maps over
    // the cache regions, 128-byte swizzle). In the reuse variant the gather
    // warps issue every tile instead (see below) and this warp idles.
    if (!GATHER && lane == 0) {
      if (g.n_r > 0) prefetch_tmap(&a.tcr);
      if (g.n_s > 0) prefetch_tmap(&a.tcs);
      int it = 0;
      bool ok = true;
      long long off = first_off;
      for (int id = first_id; id < n_items && off < end && ok; ++id) {
        const dec::Span sp = dec::item_span(a, id, ls, off, start, end);
        const int lo = sp.lo, hi = sp.hi;
        off += sp.units;
        if (lo >= hi) continue;
        const int b = id / HK, k = id - b * HK;
        const bool strm = k >= g.n_r;
        const int region = strm ? b * g.n_s + (k - g.n_r) : b * g.n_r + k;
        const CUtensorMap* map = strm ? &a.tcs : &a.tcr;
        for (int row0 = lo; row0 < hi; row0 += kBN, ++it) {
          const int st = it % kNS;
          if (it >= kNS && !wait_bar(&empty[st], ((it / kNS) & 1) ^ 1, a.err, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[st], kStage);
          uint8_t* dst = sKV + st * kStage;
#pragma unroll
          for (int sel = 0; sel < 2; ++sel)
#pragma unroll
            for (int db = 0; db < 2; ++db)
              tma_load_4d(dst + sel * kTile + db * kBox, map, db * 64, row0, sel, region, &full[st]);
        }
      }
      // every issued copy lands before the CTA can exit
      for (int j = it > kNS ? it - kNS : 0; j < it; ++j) drain_wait(&full[j % kNS], (j / kNS) & 1, a.err);
    }
    __syncwarp();
  } else if (GATHER && warp >= 6) {
    // ------------------------------------------------------------ gatherers
    // The reuse variant's GW gather warps issue every tile of the CTA's
    // range, each of them waiting for every tile's stage to be free, in
    // order (an mbarrier parity wait is only sound within one phase of the
    // barrier, so no waiter may skip tiles). Contiguous (streaming) tiles:
    // lane 0 of warp 6 loads them with the TMA onto full[st]. Retrieval
    // items: gather warp w copies rows RPW w .. RPW w + RPW - 1 of each
    // 128-row tile of borrowed positions, one row per instruction (lanes
    // 0-15 the 16 chunks of its K row, lanes 16-31 those of its V row) with
    // 16-byte cp.async copies into the swizzled layout the MMAs read, and the
    // copies complete on gfull[st]; the new token's row (position t, not in
    // the cache yet) comes from the step's input. Lane j < RPW holds the
    // index of row RPW w + j, loaded two tiles ahead into one of two
    // registers that alternate between tiles (a register copy of an
    // in-flight load would wait for it). Row gathers through the TMA
    // (tile::gather4 or bulk row copies) ran at about 15 GB/s per SM;
    // cp.async copies scale with the issuing warps.
    const int gw = warp - 6;
    const int half = lane >> 4, ch = lane & 15;
    const uint32_t dst_lane = half * kTile + (ch >> 3) * kBox;
    const uint32_t swz = ch & 7;
    const bool loader = gw == 0 && lane == 0;  // issues the TMA tiles
    if (loader && g.n_s > 0) prefetch_tmap(&a.tcs);
    int it = 0;
    bool ok = true;
    uint32_t fpar = 0;  // loader: bit st, parity of stage st's next full[] phase
    uint32_t mine = 0;  // loader: bit st, stage st's latest tile came through the TMA
    auto stage_free = [&](int st) -> bool {  // warp-uniform
      int go = 1;
      if (lane == 0 && it >= kNS && !wait_bar(&empty[st], ((it / kNS) & 1) ^ 1, a.err, abort_flag)) go = 0;
      return __shfl_sync(0xffffffffu, go, 0) != 0;
    };
    long long off = first_off;
    for (int id = first_id; id < n_items && off < end && ok; ++id) {
      const dec::Span sp = dec::item_span(a, id, ls, off, start, end);
      const int lo = sp.lo, hi = sp.hi;
      off += sp.units;
      if (lo >= hi) continue;
      const int b = id / HK, k = id - b * HK;
      if (k >= g.n_r) {
        const int region = b * g.n_s + (k - g.n_r);
        for (int row0 = lo; row0 < hi; row0 += kBN, ++it) {
          const int st = it % kNS;
          if (!stage_free(st)) {
            ok = false;
            break;
          }
          if (loader) {
            mbar_arrive_expect_tx(&full[st], kStage);
            uint8_t* dst = sKV + st * kStage;
#pragma unroll
            for (int sel = 0; sel < 2; ++sel)
#pragma unroll
              for (int db = 0; db < 2; ++db)
                tma_load_4d(dst + sel * kTile + db * kBox, &a.tcs, db * 64, row0, sel, region, &full[st]);
            fpar ^= 1u << st;
            mine |= 1u << st;
          }
        }
        continue;
      }
      const int32_t* rowlist = a.idx + ((size_t)b * a.n_idx_groups + a.idx_map[k]) * a.top_k;
      const int t = dec::seq_len(a, b, ls);
      const bf16* src_base =
          static_cast<const bf16*>(a.kv) + g.r_region(b, k) + (half ? (size_t)g.max_seq * kD : 0) + ch * 8;
      const bf16* src_new =
          static_cast<const bf16*>(half ? a.v_new : a.k_new) + ((size_t)b * g.Hkv + g.r_head[k]) * kD + ch * 8;
      const bool idx_lane = lane < RPW;
      const int j0 = lo + RPW * gw + lane;
      int ia = idx_lane && j0 < hi ? __ldg(rowlist + j0) : 0;
      int ib = idx_lane && j0 + kBN < hi ? __ldg(rowlist + j0 + kBN) : 0;
      auto gather_tile = [&](int row0, int& buf) -> bool {
        const int my_row = idx_lane && row0 + RPW * gw + lane < hi ? min(max(buf, 0), t) : -1;
        const int jn = row0 + 2 * kBN + RPW * gw + lane;
        buf = idx_lane && jn < hi ? __ldg(rowlist + jn) : 0;
        const int st = it % kNS;
        if (!stage_free(st)) return false;
        uint8_t* tile = sKV + st * kStage + dst_lane;
#pragma unroll 8
        for (int j = 0; j < RPW; ++j) {
          const int c = __shfl_sync(0xffffffffu, my_row, j);
          const int r = RPW * gw + j;
          if (c >= 0)
            cp_async16(tile + r * 128 + ((swz ^ (uint32_t)(r & 7)) << 4),
                       c == t ? src_new : src_base + (size_t)c * kD);
        }
        cp_async_mbar_arrive(&gfull[st]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&gfull[st]);
        if (loader) mine &= ~(1u << st);
        ++it;
        return true;
      };
      for (int row0 = lo; row0 < hi; row0 += 2 * kBN) {
        if (!gather_tile(row0, ia)) {
          ok = false;
          break;
        }
        if (row0 + kBN >= hi) break;
        if (!gather_tile(row0 + kBN, ib)) {
          ok = false;
          break;
        }
      }
    }
    // every copy issued here lands before the CTA can exit: the cp.async
    // copies, and the latest TMA tile of each stage
    asm volatile("cp.async.wait_all;" ::: "memory");
    if (loader)
      for (int st = 0; st < kNS; ++st)
        if (mine & (1u << st)) drain_wait(&full[st], ((fpar >> st) & 1) ^ 1, a.err);
    __syncwarp();
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer
    const uint32_t kv_addr = smem_u32(sKV), q_addr = smem_u32(sQ), p_addr = smem_u32(sP);
    int it = 0, item_k = 0, ofw = 0;
    uint32_t fpar = 0, gpar = 0;  // bit st: parity of stage st's next full[] / gfull[] phase
    bool ok = true;
    struct Pend {
      int it, st, item;
      bool first;
    } pend{0, 0, 0, false};
    bool has_pend = false;
    auto wait_warp = [&](uint64_t* bar, uint32_t parity) {
      if (ok) ok = __all_sync(0xffffffffu, wait_bar(bar, parity, a.err, abort_flag));
    };
    // o_free phases complete once per item, in order
    auto wait_ofree = [&](int n) {
      while (ok && ofw < n) {
        wait_warp(o_free, ofw & 1);
        ++ofw;
      }
    };
    auto issue_pv = [&](const Pend& t) {
      wait_warp(&p_full[t.it & 1], (t.it >> 1) & 1);
      if (t.first && t.item >= 1) wait_ofree(t.item);  // accumulate = 0 overwrites the last item's O
      if (!ok) return;
      if (lane == 0) {
        tc_fence_after();
        const uint32_t v_addr = kv_addr + t.st * kStage + kTile;
        const uint32_t pb = p_addr + (t.it & 1) * kOpBuf;
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(v_addr + kk * 2048, kBox, 1024);
          const uint64_t bd = sdesc_sw128(pb + (kk >> 2) * (kN * 128) + (kk & 3) * 32, 16, 1024);
          tc_mma(tmem + kOcol, ad, bd, IDESC_PV, (t.first && kk == 0) ? 0u : 1u);
        }
        tc_commit(&p_free[t.it & 1]);
        tc_commit(&empty[t.st]);
      }
      __syncwarp();
    };

    // An item's global inputs (its G query rows; the new token's K and V
    // row) are fetched into registers one item ahead: under the saturated
    // HBM stream a plain load takes microseconds, which at an item switch
    // would sit between this item's last P V and the next item's first S.
    // Lane l holds 16-byte chunks l, l + 32, ... of the G x 128 query block
    // (head c / 16, chunk c % 16); lanes 0-15 the new K row's chunks, lanes
    // 16-31 the new V row's.
    constexpr int QV = (G * 16 + 31) / 32;
    uint4 qr[QV];
    uint4 nvr;
    const int ch = lane & 15;
    auto kv_head_of = [&](int id) {
      const int k = id % HK;
      return k >= g.n_r ? (int)g.s_head[k - g.n_r] : (int)g.r_head[k];
    };
    auto fetch_inputs = [&](int id) {
      const int b = id / HK, kvh = kv_head_of(id);
      const bf16* qg = static_cast<const bf16*>(a.q) + ((size_t)b * g.Hq + (size_t)kvh * G) * kD;
#pragma unroll
      for (int i = 0; i < QV; ++i) {
        const int c = lane + 32 * i;
        if (c < G * 16) qr[i] = *reinterpret_cast<const uint4*>(qg + (size_t)(c >> 4) * kD + (c & 15) * 8);
      }
      const size_t new_off = ((size_t)b * g.Hkv + kvh) * kD + ch * 8;
      nvr = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(lane < 16 ? a.k_new : a.v_new) + new_off);
    };
    int fetched = -1;  // the item whose inputs the registers hold
    if (first_id < n_items) {
      fetch_inputs(first_id);
      fetched = first_id;
    }

    long long off = first_off;
    for (int id = first_id; id < n_items && off < end && ok; ++id) {
      const dec::Span sp = dec::item_span(a, id, ls, off, start, end);
      const int lo = sp.lo, hi = sp.hi;
      off += sp.units;
      if (lo >= hi) continue;
      const int b = id / HK, k = id - b * HK;
      const bool strm = k >= g.n_r;
      const int hi_idx = strm ? k - g.n_r : k;
      const int t = dec::seq_len(a, b, ls);
      const int cap = strm ? g.S + g.W : g.max_seq;
      const int xr = strm ? (t < g.S ? t : g.S + (t - g.S) % g.W) : t;  // the new token's row
      bf16* Kc = static_cast<bf16*>(a.kv) + (strm ? g.s_region(b, hi_idx) : g.r_region(b, hi_idx));
      bf16* Vc = Kc + (size_t)cap * kD;

      // this item's Q into buffer item_k & 1, last read by the MMAs of item item_k - 2
      wait_ofree(item_k - 1);
      if (!ok) break;
      if (fetched != id) {  // an item skipped by this CTA took the prefetch
        fetch_inputs(id);
        fetched = id;
      }
      {
        uint8_t* qs = sQ + (item_k & 1) * kOpBuf;
#pragma unroll
        for (int i = 0; i < QV; ++i) {
          const int c = lane + 32 * i;
          if (c < G * 16) {
            const int h = c >> 4, cc = c & 15;
            *reinterpret_cast<uint4*>(qs + (cc >> 3) * (kN * 128) + h * 128 + (((cc & 7) ^ (h & 7)) << 4)) = qr[i];
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
      }
      const uint4 nv = nvr;
      // the next item of this CTA's range starts at its row 0
      if (off < end && id + 1 < n_items) {
        fetch_inputs(id + 1);
        fetched = id + 1;
      }

      // H2Share reuse step: this retrieval item's rows are gathered
      const bool gathered = GATHER && a.idx != nullptr && !strm;
      for (int row0 = lo; row0 < hi; row0 += kBN, ++it) {
        const int st = it % kNS;
        const int cnt = min(kBN, hi - row0);
        // a tile landed on full[st] (TMA) or gfull[st] (gather warps)
        wait_warp(gathered ? &gfull[st] : &full[st], ((gathered ? gpar : fpar) >> st) & 1);
        if (gathered)
          gpar ^= 1u << st;
        else
          fpar ^= 1u << st;
        if (!ok) break;
        auto put_new_row = [&](int r) {  // the new token's K / V chunk into tile slot r
          uint8_t* dst = sKV + st * kStage + (lane < 16 ? 0 : kTile) + (ch >> 3) * kBox + r * 128 +
                         (((ch & 7) ^ (r & 7)) << 4);
          *reinterpret_cast<uint4*>(dst) = nv;
        };
        if (gathered) {
          // the gather warps wrote this tile with cp.async (generic proxy):
          // order it before the tensor core's reads; the item's owner of row
          // 0 appends the new token
          if (row0 == 0) *reinterpret_cast<uint4*>((lane < 16 ? Kc : Vc) + (size_t)xr * kD + ch * 8) = nv;
          fence_proxy_async_smem();
          __syncwarp();
        } else if (xr >= row0 && xr < row0 + cnt) {
          put_new_row(xr - row0);
          *reinterpret_cast<uint4*>((lane < 16 ? Kc : Vc) + (size_t)xr * kD + ch * 8) = nv;  // append
          fence_proxy_async_smem();
          __syncwarp();
        }
        if (it >= 2) wait_warp(&s_free[it & 1], ((it >> 1) - 1) & 1);
        if (!ok) break;
        if (lane == 0) {
          tc_fence_after();
          const uint32_t k_addr = kv_addr + st * kStage;
          const uint32_t qb = q_addr + (item_k & 1) * kOpBuf;
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint64_t ad = sdesc_sw128(k_addr + (kk >> 2) * kBox + (kk & 3) * 32, 16, 1024);
            const uint64_t bd = sdesc_sw128(qb + (kk >> 2) * (kN * 128) + (kk & 3) * 32, 16, 1024);
            tc_mma(tmem + (it & 1) * kN, ad, bd, IDESC_S, kk > 0 ? 1u : 0u);
          }
          tc_commit(&s_full[it & 1]);
        }
        __syncwarp();
        if (has_pend) issue_pv(pend);
        pend = Pend{it, st, item_k, row0 == lo};
        has_pend = true;
        if (gathered) {
          // a gathered tile's P V goes out as soon as its P is written:
          // the next tile arrives late (random rows), and its stage is
          // freed only by this P V
          issue_pv(pend);
          has_pend = false;
        }
      }
      // Inside an item, P(j) V(j) waits behind S(j + 1) so that the softmax
      // of tile j + 1 can start meanwhile. At the item's end nothing can
      // use the next item's S before this item's O is final, and holding
      // P V back until the next item's first tile lands (a loaded-DRAM
      // round trip) would hold the epilogue and this tile's ring slot.
      if (has_pend && ok) {
        issue_pv(pend);
        has_pend = false;
      }
      ++item_k;
    }
    if (has_pend) issue_pv(pend);
    if (lane == 0) {
      tc_commit(drain);
      drain_wait(drain, 0, a.err);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    const int t = threadIdx.x;  // key of the tile / row d of O^T
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    int it = 0;
    // ok: the four warps' common verdict, only ever set at a barrier (so every
    // thread leaves the loops together); local_ok: this thread's waits since
    bool ok = true, local_ok = true;
    uint32_t fpar = 0, gpar = 0;  // bit st: parity of stage st's next full[] / gfull[] phase
    long long off = first_off;
    for (int id = first_id; id < n_items && off < end && ok; ++id) {
      const dec::Span sp = dec::item_span(a, id, ls, off, start, end);
      const int rows = sp.rows, lo = sp.lo, hi = sp.hi;
      const long long item_off = off;
      off += sp.units;
      if (lo >= hi) continue;
      const int b = id / HK, k = id - b * HK;
      const bool strm = k >= g.n_r;
      const int kvh = strm ? g.s_head[k - g.n_r] : g.r_head[k];

      float m[G], l[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
      }
      const bool gathered = GATHER && a.idx != nullptr && !strm;
      for (int row0 = lo; row0 < hi; row0 += kBN, ++it) {
        const int x = it & 1, st = it % kNS;
        const int cnt = min(kBN, hi - row0);
        const uint32_t land_par = ((gathered ? gpar : fpar) >> st) & 1;  // the phase that lands this tile
        if (gathered)
          gpar ^= 1u << st;
        else
          fpar ^= 1u << st;
        local_ok = wait_bar(&s_full[x], (it >> 1) & 1, a.err, abort_flag) && local_ok;
        tc_fence_after();
        uint32_t v[16];
        tmem_ld16(tl + x * kN, v);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[x]);
        const bool valid = t < cnt;
        float s[G];
#pragma unroll
        for (int h = 0; h < G; ++h) s[h] = valid ? __uint_as_float(v[h]) * a.scale_log2 : -INFINITY;
        if (a.scores != nullptr && !strm && valid) {
          // H2Share anchor step: this row's scores for the top-k selection
          float* sc = a.scores + ((size_t)(b * g.n_r + k) * G) * a.score_stride + row0 + t;
#pragma unroll
          for (int h = 0; h < G; ++h) sc[(size_t)h * a.score_stride] = s[h];
        }

        // per-head maximum over the tile: each warp, then the four warps
        float* rx = red + x * 64;
        float wm = -INFINITY;
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float r = warp_max(s[h]);
          wm = (lane == h) ? r : wm;
        }
        if (lane < G) rx[warp * 16 + lane] = wm;
        ok = named_barrier_and(1, kSoftmaxThreads, local_ok);
        if (!ok) break;
        bool resc = false;
        float alpha[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float tm = fmaxf(fmax3f(rx[h], rx[16 + h], rx[32 + h]), rx[48 + h]);
          const float mn = fmaxf(m[h], tm);
          alpha[h] = 1.f;
          if (mn > m[h] + kRescaleThreshold) {
            alpha[h] = (m[h] == -INFINITY) ? 0.f : fast_exp2(m[h] - mn);
            m[h] = mn;
            l[h] *= alpha[h];
            resc = true;
          }
        }
        // P buffer x is free once O += P(it - 2) V is done
        if (it >= 2) local_ok = wait_bar(&p_free[x], ((it >> 1) - 1) & 1, a.err, abort_flag) && local_ok;
        if (resc && row0 != lo) {
          // rescale row t of O^T; O += P(it - 1) V must have landed first
          local_ok = wait_bar(&p_free[x ^ 1], ((it - 1) >> 1) & 1, a.err, abort_flag) && local_ok;
          tc_fence_after();
          uint32_t o[16];
          tmem_ld16(tl + kOcol, o);
          tmem_ld_wait();
#pragma unroll
          for (int h = 0; h < G; ++h) o[h] = __float_as_uint(__uint_as_float(o[h]) * alpha[h]);
          tmem_st16(tl + kOcol, o);
          tmem_st_wait();
        }
        float pr[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
          pr[h] = valid ? fast_exp2(s[h] - m[h]) : 0.f;
          l[h] += pr[h];
        }
        if (!valid) {
          // the tile has landed (its S is complete); zero V row t
          wait_bar(gathered ? &gfull[st] : &full[st], land_par, a.err, abort_flag);
          uint8_t* vr = sKV + st * kStage + kTile + t * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            reinterpret_cast<uint4*>(vr)[c] = make_uint4(0, 0, 0, 0);
            reinterpret_cast<uint4*>(vr + kBox)[c] = make_uint4(0, 0, 0, 0);
          }
        }
        // P^T row t -> column t of the K-major [16 heads][128 keys] buffer
        uint8_t* pb = sP + x * kOpBuf + (t >> 6) * (kN * 128) + (t & 7) * 2;
        const int j = (t & 63) >> 3;
#pragma unroll
        for (int h = 0; h < G; ++h)
          *reinterpret_cast<bf16*>(pb + h * 128 + ((j ^ (h & 7)) << 4)) = __float2bfloat16_rn(pr[h]);
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0 && !(it == 0 && p == a.stall_cta)) mbar_arrive(&p_full[x]);
      }
      if (!ok) break;

      // ---- the item's state: O^T row t, m (uniform), l summed over the keys
      const int last = it - 1;
      local_ok = wait_bar(&p_free[last & 1], (last >> 1) & 1, a.err, abort_flag) && local_ok;
      tc_fence_after();
      uint32_t o[16];
      tmem_ld16(tl + kOcol, o);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_free);
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float v = l[h];
#pragma unroll
        for (int msk = 16; msk >= 1; msk >>= 1) v += __shfl_xor_sync(0xffffffffu, v, msk);
        if (lane == 0) lsum[warp * 16 + h] = v;
      }
      ok = named_barrier_and(1, kSoftmaxThreads, local_ok);
      if (!ok) break;
      float L[G];
#pragma unroll
      for (int h = 0; h < G; ++h) L[h] = (lsum[h] + lsum[16 + h]) + (lsum[32 + h] + lsum[48 + h]);

      const long long row_off = item_off + sp.cost;  // unit of the item's row 0
      const int f = dec::cta_of(row_off, total, P);
      const int lst = dec::cta_of(row_off + (long long)(rows - 1) * sp.w, total, P);
      bf16* outp = static_cast<bf16*>(a.out) + ((size_t)b * g.Hq + (size_t)kvh * G) * kD;
      float2* st = (a.scores != nullptr && !strm) ? a.score_stats + (size_t)(b * g.n_r + k) * G : nullptr;
      if (f == lst) {
#pragma unroll
        for (int h = 0; h < G; ++h) outp[h * kD + t] = __float2bfloat16_rn(__uint_as_float(o[h]) / L[h]);
        if (st != nullptr && t < G) {
          float mt = m[0], lt = L[0];
#pragma unroll
          for (int h = 1; h < G; ++h) {
            mt = (t == h) ? m[h] : mt;
            lt = (t == h) ? L[h] : lt;
          }
          st[t] = make_float2(mt, lt);
        }
      } else {
        float* pbase = dec::partial_slot(a, p, p == f ? 1 : 0, G, kD);
#pragma unroll
        for (int h = 0; h < G; ++h) __stcg(pbase + h * kD + t, __uint_as_float(o[h]));
        float mt = m[0], lt = L[0];
#pragma unroll
        for (int h = 1; h < G; ++h) {
          mt = (t == h) ? m[h] : mt;
          lt = (t == h) ? L[h] : lt;
        }
        if (t < G) {
          __stcg(pbase + G * kD + t, mt);
          __stcg(pbase + G * kD + G + t, lt);
        }
        dec::merge_item<G, kD, kSoftmaxThreads, true>(a, p, f, lst, id, outp, ms, sh32 + 1, st);
      }
      named_barrier_sync(1, kSoftmaxThreads);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 5) tmem_dealloc(tmem, kTmemCols);
  if (threadIdx.x == 0) dec::finish_launch(a, ls);
}

template <int G, bool GATHER>
cudaError_t launch_g(const DecodeArgs& a, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(decode_tc_kernel<G, GATHER>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  // programmatic stream serialization: the kernel waits for the previous
  // work on the stream itself (griddepcontrol.wait) after its prologue
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_ctas);
  cfg.blockDim = dim3(kThreads + 32 * gather_warps(G, GATHER));
  cfg.dynamicSmemBytes = SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_tc_kernel<G, GATHER>, a);
}

}  // namespace

bool decode_uses_tc(int D, int G) { return D == kD && ((G >= 1 && G <= 8) || G == 16); }

int decode_tc_item_cost(long long total_rows, int n_ctas, int num_sms) {
  if (total_rows >= kItemCostMaxShare * n_ctas) return 0;
  return n_ctas < num_sms ? kItemCostFewCtas : kItemCost;
}

void reuse_tc_weights(int G, int* gather_w, int* ring_w) {
  (void)G;
  *gather_w = 3;
  *ring_w = 2;
}

// One CTA per SM; small steps use fewer, at least 512 rows each.
// At least 512 rows (four tiles) per CTA, so that small steps keep few
// partials per item (an item spread over more than kGroup CTAs needs the
// second merge level); once that fills half the GPU, every SM streams.
int decode_tc_ctas(long long total_rows, int num_sms) {
  const long long by_rows = (total_rows + 511) / 512;
  long long p = by_rows >= num_sms / 2 ? num_sms : by_rows;
  return p < 1 ? 1 : (int)p;
}

template <bool GATHER>
cudaError_t launch_tc(const DecodeArgs& a, cudaStream_t s) {
  switch (a.geom.G) {
    case 1: return launch_g<1, GATHER>(a, s);
    case 2: return launch_g<2, GATHER>(a, s);
    case 3: return launch_g<3, GATHER>(a, s);
    case 4: return launch_g<4, GATHER>(a, s);
    case 5: return launch_g<5, GATHER>(a, s);
    case 6: return launch_g<6, GATHER>(a, s);
    case 7: return launch_g<7, GATHER>(a, s);
    case 8: return launch_g<8, GATHER>(a, s);
    case 16: return launch_g<16, GATHER>(a, s);
  }
  return cudaErrorInvalidValue;
}

// The reuse step (a.idx set) launches the variant with gather warps.
cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t s) {
  return a.idx != nullptr ? launch_tc<true>(a, s) : launch_tc<false>(a, s);
}

}  // namespace aoh
