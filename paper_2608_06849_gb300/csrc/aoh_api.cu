// Host runtime behind include/aoh.h: argument validation, cache layout,
// split-KV scheduling and kernel launches on the caller's stream.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "../../include/aoh.h"
#include "internal.h"

using namespace aoh;

namespace {

thread_local std::string g_last_error;

aoh_status fail(aoh_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

aoh_status cuda_fail(cudaError_t e, const char* what) {
  return fail(AOH_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Validates cfg + labels; fills n_r / n_s. Returns AOH_OK or an error.
aoh_status check_config(const aoh_config* cfg, const uint8_t* labels, int* n_r, int* n_s) {
  if (!cfg) return fail(AOH_ERR_INVALID, "cfg is NULL");
  if (!labels) return fail(AOH_ERR_INVALID, "head_labels is NULL");
  const aoh_config& c = *cfg;
  if (c.batch < 1 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.max_seq < 1)
    return fail(AOH_ERR_INVALID, "batch, n_q_heads, n_kv_heads and max_seq must be >= 1");
  if (c.n_kv_heads > kMaxKvHeads) return fail(AOH_ERR_UNSUPPORTED, "n_kv_heads > %d", kMaxKvHeads);
  if (c.n_q_heads % c.n_kv_heads) return fail(AOH_ERR_INVALID, "n_q_heads must be a multiple of n_kv_heads");
  if (c.d_head != 64 && c.d_head != 128) return fail(AOH_ERR_UNSUPPORTED, "d_head must be 64 or 128");
  if (c.sink < 0 || c.window < 1) return fail(AOH_ERR_INVALID, "need sink >= 0 and window >= 1");
  if (c.chunk < 0) return fail(AOH_ERR_INVALID, "chunk must be >= 0");
  int r = 0, s = 0;
  for (int h = 0; h < c.n_kv_heads; ++h) {
    if (labels[h] == AOH_RETRIEVAL)
      ++r;
    else if (labels[h] == AOH_STREAMING)
      ++s;
    else
      return fail(AOH_ERR_INVALID, "head_labels[%d] = %d is neither retrieval (0) nor streaming (1)", h,
                  (int)labels[h]);
  }
  *n_r = r;
  *n_s = s;
  return AOH_OK;
}

// Prefill work: one item per (b, query head, 128-row query tile), with the
// number of 128-key tiles it visits as its cost; heaviest first so the
// hardware block scheduler fills the machine longest-processing-time first.
std::vector<int4> prefill_schedule(const CacheGeom& g, const std::vector<int32_t>& base,
                                   const std::vector<int32_t>& lens) {
  constexpr int BM = 256, BN = 128;
  std::vector<int4> items;
  for (int b = 0; b < g.B; ++b) {
    for (int h = 0; h < g.Hq; ++h) {
      const bool streaming = g.kind[h / g.G] != 0;
      const int Lb = base[b];
      const int n_c = Lb == 0 ? 0 : ((streaming ? std::min(Lb, g.S + g.W) : Lb) + BN - 1) / BN;
      const int S_rel = g.S - Lb;
      for (int q0 = 0; q0 < lens[b]; q0 += BM) {
        const int q_end = std::min(q0 + BM, (int)lens[b]);
        int n;
        if (!streaming) {
          n = (q_end + BN - 1) / BN;
        } else {
          const int a_end = (std::min(std::max(S_rel, 0), q_end) + BN - 1) / BN;
          const int c_begin = std::max(a_end, std::max(0, g.wstart(q0)) / BN);
          const int c_end = std::max(c_begin, (q_end + BN - 1) / BN);
          n = a_end + (c_end - c_begin);
        }
        items.push_back(make_int4(b, h, q0, n_c + n));
      }
    }
  }
  std::stable_sort(items.begin(), items.end(), [](const int4& x, const int4& y) { return x.w > y.w; });
  return items;
}

size_t bytes_for(const aoh_config& c, int n_r, int n_s) {
  const size_t tokens = (size_t)n_r * c.max_seq + (size_t)n_s * (size_t)(c.sink + c.window);
  return (size_t)c.batch * tokens * c.d_head * 2 * 2;
}

}  // namespace

void aoh::record_error(const char* msg) { g_last_error = msg; }

struct aoh_cache {
  CUtensorMap tcr, tcs;  // cache regions for TMA (built once: the buffer does not move)
  aoh_config cfg;
  CacheGeom geom;
  std::vector<uint8_t> labels;
  void* kv = nullptr;
  size_t kv_bytes = 0;
  std::vector<int32_t> lens;  // host mirror of the device lengths
  int device = 0;
  int num_sms = 0;
  // device metadata (one allocation)
  void* meta = nullptr;
  int32_t* d_lens = nullptr;
  int32_t* d_chunk = nullptr;  // rows of the current prefill chunk
  uint32_t* d_counters = nullptr;
  uint32_t* d_gcounters = nullptr;
  uint32_t* d_done = nullptr;
  uint32_t* d_err = nullptr;
  float* d_partials = nullptr;
  // prefill work list (device), grown on demand
  int4* d_work = nullptr;
  size_t work_cap = 0;
  // H2Share anchor workspace (scores, head states, importance overflow),
  // allocated on first use
  float* d_h2 = nullptr;
};

namespace {

// Grow the prefill work list to at least n items (cudaMalloc, which
// synchronises the device).
cudaError_t reserve_work(aoh_cache* h, size_t n) {
  if (n <= h->work_cap) return cudaSuccess;
  if (h->d_work) cudaFree(h->d_work);
  h->d_work = nullptr;
  h->work_cap = 0;
  cudaError_t e = cudaMalloc(&h->d_work, n * sizeof(int4));
  if (e == cudaSuccess) h->work_cap = n;
  return e;
}

// Work items of a prefill call whose chunks hold up to `tokens` rows: one per
// (sequence, query head, 256-row pair of query tiles).
size_t work_items_for(const CacheGeom& g, long long tokens) {
  return (size_t)g.B * g.Hq * (size_t)((tokens + 255) / 256);
}

// The H2Share anchor workspace (once per handle; cudaMalloc).
cudaError_t reserve_h2(aoh_cache* h) {
  const CacheGeom& g = h->geom;
  if (g.n_r == 0 || h->d_h2) return cudaSuccess;
  // scores [B][n_r][G][max_seq padded to 4], head states, importance overflow
  cudaError_t e = cudaMalloc(&h->d_h2, h2_workspace_floats(g.B, g.n_r, g.G, g.max_seq) * sizeof(float));
  if (e != cudaSuccess) h->d_h2 = nullptr;
  return e;
}

}  // namespace

extern "C" {

int32_t aoh_version(void) { return 102; }

const char* aoh_last_error(void) { return g_last_error.c_str(); }

size_t aoh_cache_bytes(const aoh_config* cfg, const uint8_t* head_labels) {
  int n_r, n_s;
  if (check_config(cfg, head_labels, &n_r, &n_s) != AOH_OK) return 0;
  return bytes_for(*cfg, n_r, n_s);
}

aoh_status aoh_cache_init(const aoh_config* cfg, const uint8_t* head_labels, void* kv_buffer,
                          size_t kv_buffer_bytes, aoh_cache** out) {
  if (!out) return fail(AOH_ERR_INVALID, "out is NULL");
  *out = nullptr;
  int n_r, n_s;
  aoh_status st = check_config(cfg, head_labels, &n_r, &n_s);
  if (st != AOH_OK) return st;
  const aoh_config& c = *cfg;
  const int G = c.n_q_heads / c.n_kv_heads;
  if (!decode_supported(c.d_head, G))
    return fail(AOH_ERR_UNSUPPORTED, "group size %d with d_head %d is not compiled", G, c.d_head);
  if (!kv_buffer) return fail(AOH_ERR_INVALID, "kv_buffer is NULL");
  if (!aligned(kv_buffer, 256)) return fail(AOH_ERR_INVALID, "kv_buffer must be 256-byte aligned");
  const size_t need = bytes_for(c, n_r, n_s);
  if (kv_buffer_bytes < need)
    return fail(AOH_ERR_CAPACITY, "kv_buffer has %zu bytes, the cache needs %zu", kv_buffer_bytes, need);

  aoh_cache* h = new aoh_cache();
  h->cfg = c;
  h->labels.assign(head_labels, head_labels + c.n_kv_heads);
  h->kv = kv_buffer;
  h->kv_bytes = need;
  h->lens.assign(c.batch, 0);
  CacheGeom& g = h->geom;
  g.B = c.batch;
  g.Hq = c.n_q_heads;
  g.Hkv = c.n_kv_heads;
  g.D = c.d_head;
  g.G = G;
  g.max_seq = c.max_seq;
  g.S = c.sink;
  g.W = c.window;
  g.K = c.chunk;
  g.n_r = n_r;
  g.n_s = n_s;
  int ir = 0, is = 0;
  for (int k = 0; k < c.n_kv_heads; ++k) {
    g.kind[k] = head_labels[k];
    if (head_labels[k] == AOH_RETRIEVAL) {
      g.idx[k] = (uint8_t)ir;
      g.r_head[ir++] = (uint8_t)k;
    } else {
      g.idx[k] = (uint8_t)is;
      g.s_head[is++] = (uint8_t)k;
    }
  }

  cudaError_t e = cudaGetDevice(&h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (e != cudaSuccess) {
    delete h;
    return cuda_fail(e, "cudaGetDevice");
  }
  const size_t n_lens = ((size_t)c.batch + 63) / 64 * 64;
  const size_t n_cnt = ((size_t)c.batch * c.n_kv_heads + 63) / 64 * 64;
  const size_t n_part = decode_partial_floats(2 * h->num_sms, G, c.d_head);
  const size_t n_gcnt = ((size_t)4 * h->num_sms + 63) / 64 * 64;
  const size_t meta_bytes = (2 * n_lens + n_cnt + n_gcnt + 64) * 4 + n_part * 4;
  e = cudaMalloc(&h->meta, meta_bytes);
  if (e == cudaSuccess) e = cudaMemset(h->meta, 0, meta_bytes);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    if (h->meta) cudaFree(h->meta);
    delete h;
    return cuda_fail(e, "metadata allocation");
  }
  uint32_t* base = static_cast<uint32_t*>(h->meta);
  h->d_lens = reinterpret_cast<int32_t*>(base);
  h->d_chunk = reinterpret_cast<int32_t*>(base + n_lens);
  h->d_counters = base + 2 * n_lens;
  h->d_gcounters = h->d_counters + n_cnt;
  h->d_done = h->d_gcounters + n_gcnt;
  h->d_err = h->d_done + 32;
  h->d_partials = reinterpret_cast<float*>(base + 2 * n_lens + n_cnt + n_gcnt + 64);
  if (!make_cache_region_maps(&h->tcr, &h->tcs, h->geom, h->kv)) {
    cudaFree(h->meta);
    delete h;
    return fail(AOH_ERR_CUDA, "cuTensorMapEncodeTiled failed for the cache regions");
  }
  // the prefill work list for the longest chunk a retrieval head can take
  // (max_seq tokens), so that prefill calls within it allocate nothing
  e = reserve_work(h, work_items_for(h->geom, c.max_seq));
  if (e != cudaSuccess) {
    cudaFree(h->meta);
    delete h;
    return cuda_fail(e, "work list allocation");
  }
  *out = h;
  return AOH_OK;
}

aoh_status aoh_cache_reserve(aoh_cache* cache, int32_t max_tokens, int32_t anchor_workspace) {
  if (!cache) return fail(AOH_ERR_INVALID, "cache is NULL");
  if (max_tokens < 0) return fail(AOH_ERR_INVALID, "max_tokens must be >= 0");
  cudaError_t e = reserve_work(cache, work_items_for(cache->geom, max_tokens));
  if (e != cudaSuccess) return cuda_fail(e, "work list allocation");
  if (anchor_workspace) {
    if (!decode_uses_tc(cache->geom.D, cache->geom.G))
      return fail(AOH_ERR_UNSUPPORTED, "the anchor step needs the d_head 128 tensor-core decode");
    e = reserve_h2(cache);
    if (e != cudaSuccess) return cuda_fail(e, "anchor workspace allocation");
  }
  return AOH_OK;
}

void aoh_cache_destroy(aoh_cache* cache) {
  if (!cache) return;
  if (cache->meta) cudaFree(cache->meta);
  if (cache->d_work) cudaFree(cache->d_work);
  if (cache->d_h2) cudaFree(cache->d_h2);
  delete cache;
}

aoh_status aoh_cache_lens(const aoh_cache* cache, int32_t* lens_out) {
  if (!cache || !lens_out) return fail(AOH_ERR_INVALID, "NULL argument");
  std::copy(cache->lens.begin(), cache->lens.end(), lens_out);
  return AOH_OK;
}

aoh_status aoh_cache_region(const aoh_cache* cache, int32_t b, int32_t kv_head, size_t* k_offset,
                            size_t* v_offset, int32_t* capacity) {
  if (!cache || !k_offset || !v_offset || !capacity) return fail(AOH_ERR_INVALID, "NULL argument");
  const CacheGeom& g = cache->geom;
  if (b < 0 || b >= g.B || kv_head < 0 || kv_head >= g.Hkv) return fail(AOH_ERR_INVALID, "b or kv_head out of range");
  const size_t elem = g.region(b, kv_head);
  *capacity = g.capacity(kv_head);
  *k_offset = elem * 2;
  *v_offset = (elem + (size_t)(*capacity) * g.D) * 2;
  return AOH_OK;
}

aoh_status aoh_cache_reset(aoh_cache* cache, void* stream) {
  if (!cache) return fail(AOH_ERR_INVALID, "cache is NULL");
  std::fill(cache->lens.begin(), cache->lens.end(), 0);
  cudaError_t e = cudaMemsetAsync(cache->d_lens, 0, sizeof(int32_t) * cache->geom.B, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
  return AOH_OK;
}

aoh_status aoh_cache_check(aoh_cache* cache, void* stream) {
  if (!cache) return fail(AOH_ERR_INVALID, "cache is NULL");
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  uint32_t err = 0;
  e = cudaMemcpy(&err, cache->d_err, sizeof(err), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
  if (err) {
    const uint32_t zero = 0;
    cudaMemcpy(cache->d_err, &zero, sizeof(zero), cudaMemcpyHostToDevice);
    if (err & kErrTimeout) return fail(AOH_ERR_TIMEOUT, "a kernel's bounded wait ran out (error word 0x%x)", err);
    return fail(AOH_ERR_CAPACITY, "a decode step found a sequence already holding max_seq tokens (error word 0x%x)",
                err);
  }
  return AOH_OK;
}

aoh_status aoh_cache_selftest_wait(aoh_cache* cache, int64_t limit_ns, int64_t* elapsed_ns, void* stream) {
  if (!cache) return fail(AOH_ERR_INVALID, "cache is NULL");
  if (limit_ns < 1000000 || limit_ns > 2000000000LL)
    return fail(AOH_ERR_INVALID, "limit_ns must be in [1 ms, 2 s]");
  cudaStream_t s = (cudaStream_t)stream;
  // the elapsed time is staged in the metadata block's spare word after the error word
  unsigned long long* d_elapsed = reinterpret_cast<unsigned long long*>(cache->d_err + 8);
  cudaError_t e = launch_wait_selftest(cache->d_err, (uint64_t)limit_ns, d_elapsed, s);
  if (e != cudaSuccess) return cuda_fail(e, "self-test kernel launch");
  unsigned long long el = 0;
  e = cudaMemcpyAsync(&el, d_elapsed, sizeof(el), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "self-test read back");
  if (elapsed_ns) *elapsed_ns = (int64_t)el;
  return AOH_OK;
}

aoh_status aoh_prefill(const void* q, const void* k, const void* v, int32_t T, const int32_t* seq_lens,
                       aoh_cache* cache, void* out, void* stream) {
  if (!cache) return fail(AOH_ERR_INVALID, "cache is NULL");
  if (!k || !v) return fail(AOH_ERR_INVALID, "k and v must not be NULL");
  if (out && !q) return fail(AOH_ERR_INVALID, "q must not be NULL when out is given");
  if (!aligned(k, 16) || !aligned(v, 16) || (q && !aligned(q, 16)) || (out && !aligned(out, 16)))
    return fail(AOH_ERR_INVALID, "q, k, v and out must be 16-byte aligned");
  const CacheGeom& g = cache->geom;
  if (T < 1) return fail(AOH_ERR_INVALID, "T must be >= 1");
  std::vector<int32_t> clen(g.B, T);
  if (seq_lens) {
    for (int b = 0; b < g.B; ++b) {
      if (seq_lens[b] < 1 || seq_lens[b] > T)
        return fail(AOH_ERR_INVALID, "seq_lens[%d] = %d is outside [1, T]", b, seq_lens[b]);
      clen[b] = seq_lens[b];
    }
  }
  const std::vector<int32_t> base = cache->lens;
  if (g.K > 0)
    for (int b = 0; b < g.B; ++b)
      if (base[b] % g.K)
        return fail(AOH_ERR_INVALID, "sequence %d holds %d tokens, not a multiple of chunk %d", b, base[b], g.K);
  std::vector<int32_t> lens(g.B);
  bool chunked = false;
  for (int b = 0; b < g.B; ++b) {
    lens[b] = base[b] + clen[b];
    chunked |= base[b] > 0;
    if (g.n_r > 0 && lens[b] > g.max_seq)
      return fail(AOH_ERR_CAPACITY, "sequence %d would hold %d tokens; max_seq is %d", b, lens[b], g.max_seq);
  }
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(cache->d_chunk, clen.data(), sizeof(int32_t) * g.B, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(chunk lengths)");

  // attention first: a chunk's own writes to a streaming ring would overwrite
  // positions its rows still read
  if (out) {
    const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)g.D));
    std::vector<int4> items = prefill_schedule(g, base, clen);
    e = reserve_work(cache, items.size());
    if (e != cudaSuccess) return cuda_fail(e, "work list allocation");
    e = cudaMemcpyAsync(cache->d_work, items.data(), items.size() * sizeof(int4), cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(work)");
    PrefillTcArgs pa;
    memset(&pa, 0, sizeof(pa));
    pa.geom = g;
    pa.out = out;
    pa.lens = cache->d_chunk;
    pa.base = cache->d_lens;
    pa.work = cache->d_work;
    pa.err = cache->d_err;
    pa.T = T;
    pa.scale_log2 = scale_log2;
    if (!prefill_tc_make_maps(&pa, q, k, v, g.B, T))
      return fail(AOH_ERR_CUDA, "cuTensorMapEncodeTiled failed for q/k/v");
    if (chunked && !prefill_tc_make_cache_maps(&pa, cache->kv))
      return fail(AOH_ERR_CUDA, "cuTensorMapEncodeTiled failed for the cache");
    e = launch_prefill_tc(pa, (int)items.size(), s);
    if (e != cudaSuccess) return cuda_fail(e, "prefill kernel launch");
  }

  AppendArgs ap;
  ap.geom = g;
  ap.k = k;
  ap.v = v;
  ap.kv = cache->kv;
  ap.lens = cache->d_chunk;
  ap.base = cache->d_lens;
  ap.T = T;
  e = launch_append(ap, s);
  if (e != cudaSuccess) return cuda_fail(e, "append kernel launch");
  e = launch_lens_add(cache->d_lens, cache->d_chunk, g.B, s);
  if (e != cudaSuccess) return cuda_fail(e, "length update launch");
  cache->lens = lens;
  return AOH_OK;
}

}  // extern "C"

namespace {

// Host checks shared by the decode entry points; fills `a` for the step and
// the step's total rows (every retrieval row; ring rows of streaming heads).
aoh_status prepare_decode(const void* q, const void* k_new, const void* v_new, aoh_cache* cache, void* out,
                          DecodeArgs& a, long long& total) {
  if (!cache) return fail(AOH_ERR_INVALID, "cache is NULL");
  if (!q || !k_new || !v_new || !out) return fail(AOH_ERR_INVALID, "q, k_new, v_new and out must not be NULL");
  if (!aligned(q, 16) || !aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(out, 16))
    return fail(AOH_ERR_INVALID, "q, k_new, v_new and out must be 16-byte aligned");
  const CacheGeom& g = cache->geom;
  total = 0;
  for (int b = 0; b < g.B; ++b) {
    if (g.n_r > 0 && cache->lens[b] + 1 > g.max_seq)
      return fail(AOH_ERR_CAPACITY, "sequence %d holds %d tokens; max_seq is %d", b, cache->lens[b], g.max_seq);
    const long long t1 = cache->lens[b] + 1;
    total += g.n_r * t1 + g.n_s * std::min<long long>(t1, g.S + g.W);
  }
  a.tcr = cache->tcr;
  a.tcs = cache->tcs;
  a.geom = g;
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  a.out = out;
  a.kv = cache->kv;
  a.lens = cache->d_lens;
  a.partials = cache->d_partials;
  a.counters = cache->d_counters;
  a.gcounters = cache->d_gcounters;
  a.done = cache->d_done;
  a.err = cache->d_err;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)g.D));
  return AOH_OK;
}

}  // namespace

extern "C" {

aoh_status aoh_decode_step(const void* q, const void* k_new, const void* v_new, aoh_cache* cache, void* out,
                           void* stream) {
  DecodeArgs a;
  long long total = 0;
  const aoh_status st = prepare_decode(q, k_new, v_new, cache, out, a, total);
  if (st != AOH_OK) return st;
  const CacheGeom& g = cache->geom;
  a.n_ctas = decode_ctas(total, cache->num_sms, g.D, g.G);
  if (decode_uses_tc(g.D, g.G)) a.item_cost = decode_tc_item_cost(total, a.n_ctas, cache->num_sms);
  cudaError_t e = launch_decode(a, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "decode kernel launch");
  for (int b = 0; b < g.B; ++b) cache->lens[b] += 1;
  return AOH_OK;
}

aoh_status aoh_decode_step_anchor(const void* q, const void* k_new, const void* v_new, aoh_cache* cache, void* out,
                                  int32_t top_k, int32_t* indices, void* stream) {
  DecodeArgs a;
  long long total = 0;
  const aoh_status st = prepare_decode(q, k_new, v_new, cache, out, a, total);
  if (st != AOH_OK) return st;
  const CacheGeom& g = cache->geom;
  if (top_k < 1) return fail(AOH_ERR_INVALID, "top_k must be >= 1");
  if (g.n_r > 0 && !indices) return fail(AOH_ERR_INVALID, "indices must not be NULL");
  if (!decode_uses_tc(g.D, g.G))
    return fail(AOH_ERR_UNSUPPORTED, "the anchor step needs the d_head 128 tensor-core decode");
  if (g.n_r > 0 && !cache->d_h2) {
    cudaError_t e = reserve_h2(cache);
    if (e != cudaSuccess) return cuda_fail(e, "anchor workspace allocation");
  }
  if (g.n_r > 0) h2_decode_outputs(cache->d_h2, g.B, g.n_r, g.G, g.max_seq, &a.scores, &a.score_stride, &a.score_stats);
  a.n_ctas = decode_ctas(total, cache->num_sms, g.D, g.G);
  a.item_cost = decode_tc_item_cost(total, a.n_ctas, cache->num_sms);
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = launch_decode(a, s);
  if (e != cudaSuccess) return cuda_fail(e, "decode kernel launch");
  for (int b = 0; b < g.B; ++b) cache->lens[b] += 1;
  if (g.n_r > 0) {
    e = launch_h2_topk(cache->d_h2, g.max_seq, cache->d_lens, g.B, g.n_r, g.G, top_k, indices, s);
    if (e != cudaSuccess) return cuda_fail(e, "top-k kernel launch");
  }
  return AOH_OK;
}

aoh_status aoh_decode_step_reuse(const void* q, const void* k_new, const void* v_new, aoh_cache* cache, void* out,
                                 const int32_t* indices, int32_t n_anchor_groups, int32_t top_k,
                                 const int32_t* group_map, void* stream) {
  DecodeArgs a;
  long long total = 0;
  const aoh_status st = prepare_decode(q, k_new, v_new, cache, out, a, total);
  if (st != AOH_OK) return st;
  const CacheGeom& g = cache->geom;
  // d_head 128: the tcgen05 kernel's gather warps copy the borrowed rows, a
  // gathered row weighing gather_w / ring_w contiguous rows in the CTA split
  const bool tc = decode_uses_tc(g.D, g.G);
  if (!tc && !decode_cc_supported(g.D, g.G))
    return fail(AOH_ERR_UNSUPPORTED, "group size not compiled for the reuse step");
  if (top_k < 1) return fail(AOH_ERR_INVALID, "top_k must be >= 1");
  if (g.n_r > 0) {
    if (!indices || !group_map) return fail(AOH_ERR_INVALID, "indices and group_map must not be NULL");
    if (!aligned(indices, 4)) return fail(AOH_ERR_INVALID, "indices must be 4-byte aligned");
    if (n_anchor_groups < 1 || n_anchor_groups > kMaxKvHeads)
      return fail(AOH_ERR_INVALID, "n_anchor_groups must be in [1, %d]", kMaxKvHeads);
    for (int i = 0; i < g.n_r; ++i)
      if (group_map[i] < 0 || group_map[i] >= n_anchor_groups)
        return fail(AOH_ERR_INVALID, "group_map[%d] = %d is outside [0, %d)", i, group_map[i], n_anchor_groups);
    for (int i = 0; i < g.n_r; ++i) a.idx_map[i] = (uint8_t)group_map[i];
  }
  a.idx = g.n_r > 0 ? indices : nullptr;
  a.top_k = top_k;
  a.n_idx_groups = n_anchor_groups;
  if (tc) reuse_tc_weights(g.G, &a.gather_w, &a.ring_w);
  // every retrieval item now holds min(top_k, t + 1) rows
  total = 0;
  for (int b = 0; b < g.B; ++b) {
    const long long t1 = cache->lens[b] + 1;
    total += (g.n_r * std::min<long long>(t1, top_k) * a.gather_w +
              g.n_s * std::min<long long>(t1, g.S + g.W) * a.ring_w + a.ring_w - 1) / a.ring_w;
  }
  a.n_ctas = tc ? decode_tc_ctas(total, cache->num_sms) : decode_cc_ctas(total, cache->num_sms);
  cudaError_t e = tc ? launch_decode_tc(a, (cudaStream_t)stream) : launch_decode_cc(a, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "reuse decode kernel launch");
  for (int b = 0; b < g.B; ++b) cache->lens[b] += 1;
  return AOH_OK;
}

}  // extern "C"
