// A decode step for callers that cannot allocate device memory.
//
// Some callers must not allocate device memory once they are running: an
// inference server that reserves its whole memory arena at start-up and
// treats any later cudaMalloc as a failure, or a latency-critical loop where
// cudaMalloc's implicit device-wide synchronisation would stall every other
// stream. aoh_cache_init allocates a small metadata block, so those callers
// cannot use the handle API for decode. This entry point runs the same
// split-KV decode kernel, but its scratch (split partials, arrival counters,
// the error word) lives in one statically allocated device array of this
// file, sized kNoAllocScratchBytes (16 MiB + 128 KiB). Every GPU that loads the library holds
// that array until the process exits.
//
// The array's host-side name is only a stand-in for the device symbol, so the
// device address is looked up with cudaGetSymbolAddress the first time a
// device calls in (with that device current) and cached per device.
#include <math.h>
#include <stdio.h>

#include <mutex>

#include "../../include/aoh.h"
#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

constexpr size_t kNoAllocHeaderBytes = 128 * 1024;        // err, status, done, item and group counters
constexpr int kStatusWord = 16;                            // sticky status: header word 16
constexpr size_t kNoAllocPartialBytes = 16u * 1024 * 1024;  // split-KV partials
constexpr size_t kNoAllocScratchBytes = kNoAllocHeaderBytes + kNoAllocPartialBytes;
constexpr int kNoAllocMaxItems = 16320;  // B * n_kv_heads limit
constexpr int kNoAllocMaxCtas = 2048;    // decode CTAs (two group counters each)
static_assert(64 + kNoAllocMaxItems + 2 * kNoAllocMaxCtas <= (int)(kNoAllocHeaderBytes / 4), "header");
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};

aoh_status set_err(aoh_status st, const char* msg) {
  record_error(msg);
  return st;
}

}  // namespace
}  // namespace aoh

using namespace aoh;

namespace {

// The allocation-free step; stall_cta >= 0 runs the self-test (on the
// launch's last CTA).
aoh_status noalloc_step(const aoh_config* cfg, const uint8_t* head_labels, void* kv_buffer, int32_t* lens,
                        int32_t max_len, const void* q, const void* k_new, const void* v_new, void* out,
                        void* stream, int stall_cta) {
  if (!cfg || !head_labels || !kv_buffer || !lens || !q || !k_new || !v_new || !out)
    return set_err(AOH_ERR_INVALID, "aoh_decode_step_noalloc: NULL argument");
  const aoh_config& c = *cfg;
  if (c.batch < 1 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.n_kv_heads > kMaxKvHeads || c.max_seq < 1 ||
      c.n_q_heads % c.n_kv_heads || (c.d_head != 64 && c.d_head != 128) || c.sink < 0 || c.window < 1)
    return set_err(AOH_ERR_INVALID, "aoh_decode_step_noalloc: invalid config");
  const int G = c.n_q_heads / c.n_kv_heads;
  if (!decode_supported(c.d_head, G))
    return set_err(AOH_ERR_UNSUPPORTED, "aoh_decode_step_noalloc: group size not compiled");
  if (stall_cta >= 0 && !decode_uses_tc(c.d_head, G))
    return set_err(AOH_ERR_UNSUPPORTED, "aoh_decode_step_noalloc_selftest: needs the d_head 128 tensor-core decode");
  const uintptr_t al = reinterpret_cast<uintptr_t>(kv_buffer) | reinterpret_cast<uintptr_t>(q) |
                       reinterpret_cast<uintptr_t>(k_new) | reinterpret_cast<uintptr_t>(v_new) |
                       reinterpret_cast<uintptr_t>(out);
  if (al % 16 || reinterpret_cast<uintptr_t>(kv_buffer) % 256)
    return set_err(AOH_ERR_INVALID, "aoh_decode_step_noalloc: misaligned pointer");
  const int items = c.batch * c.n_kv_heads;
  if (items > kNoAllocMaxItems)
    return set_err(AOH_ERR_CAPACITY,
                   "aoh_decode_step_noalloc: batch * n_kv_heads exceeds the static scratch limit of 16320");

  CacheGeom g;
  g.B = c.batch;
  g.Hq = c.n_q_heads;
  g.Hkv = c.n_kv_heads;
  g.D = c.d_head;
  g.G = G;
  g.max_seq = c.max_seq;
  g.S = c.sink;
  g.W = c.window;
  g.K = c.chunk;
  int n_r = 0, n_s = 0;
  for (int h = 0; h < c.n_kv_heads; ++h) {
    if (head_labels[h] == AOH_RETRIEVAL) {
      g.kind[h] = 0;
      g.idx[h] = (uint8_t)n_r;
      g.r_head[n_r++] = (uint8_t)h;
    } else if (head_labels[h] == AOH_STREAMING) {
      g.kind[h] = 1;
      g.idx[h] = (uint8_t)n_s;
      g.s_head[n_s++] = (uint8_t)h;
    } else {
      return set_err(AOH_ERR_INVALID, "aoh_decode_step_noalloc: bad head label");
    }
  }
  g.n_r = n_r;
  g.n_s = n_s;
  if (max_len < 0) return set_err(AOH_ERR_INVALID, "aoh_decode_step_noalloc: max_len < 0");
  if (n_r > 0 && max_len + 1 > c.max_seq)
    return set_err(AOH_ERR_CAPACITY, "aoh_decode_step_noalloc: a retrieval head would pass max_seq");

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc: cudaGetDevice failed");
  void* scratch = nullptr;
  int num_sms = 0;
  {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_ptr[dev]) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (e != cudaSuccess) return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc: cudaGetSymbolAddress failed");
      int sms = 0;
      e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc: device query failed");
      g_num_sms[dev] = sms;
      g_scratch_ptr[dev] = p;
    }
    scratch = g_scratch_ptr[dev];
    num_sms = g_num_sms[dev];
  }
  uint32_t* header = static_cast<uint32_t*>(scratch);
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  // CTA count as the handle API computes it (from an upper bound of the rows),
  // bounded by the partial space.
  const long long t1 = (long long)max_len + 1;
  const long long win = t1 < c.sink + c.window ? t1 : c.sink + c.window;
  const long long total = (long long)c.batch * ((long long)n_r * t1 + (long long)n_s * win);
  int n_ctas = decode_ctas(total, num_sms, c.d_head, G);
  const int cap_ctas = (int)(kNoAllocPartialBytes / (decode_partial_floats(1, G, c.d_head) * 4));
  if (n_ctas > cap_ctas) n_ctas = cap_ctas;
  if (n_ctas > kNoAllocMaxCtas) n_ctas = kNoAllocMaxCtas;
  // err, done and the arrival counters start at zero: the array is
  // zero-initialised, and every launch leaves them at zero (self-cleaning,
  // timeouts included), so consecutive calls need no clearing launch and
  // each decode launch overlaps the previous one's tail (programmatic
  // dependent launch).
  DecodeArgs a;
  if (!make_cache_region_maps(&a.tcr, &a.tcs, g, kv_buffer))
    return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc: cuTensorMapEncodeTiled failed");
  a.geom = g;
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  a.out = out;
  a.kv = kv_buffer;
  a.lens = lens;
  a.err = header;
  a.done = header + 32;
  a.counters = header + 64;
  a.gcounters = header + 64 + items;
  a.partials = reinterpret_cast<float*>(static_cast<unsigned char*>(scratch) + kNoAllocHeaderBytes);
  a.n_ctas = n_ctas;
  if (decode_uses_tc(c.d_head, G)) a.item_cost = decode_tc_item_cost(total, n_ctas, num_sms);
  a.self_clean = 1;
  a.status = header + kStatusWord;
  // the self-test stalls the launch's last CTA: the step's last row is
  // always its, whereas an item charge can leave the first CTAs without rows
  a.stall_cta = stall_cta >= 0 ? n_ctas - 1 : -1;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)c.d_head));
  e = launch_decode(a, s);
  if (e != cudaSuccess) return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc: kernel launch failed");
  return AOH_OK;
}

}  // namespace

extern "C" aoh_status aoh_decode_step_noalloc(const aoh_config* cfg, const uint8_t* head_labels, void* kv_buffer,
                                              int32_t* lens, int32_t max_len, const void* q, const void* k_new,
                                              const void* v_new, void* out, void* stream) {
  return noalloc_step(cfg, head_labels, kv_buffer, lens, max_len, q, k_new, v_new, out, stream, -1);
}

extern "C" aoh_status aoh_decode_step_noalloc_selftest(const aoh_config* cfg, const uint8_t* head_labels,
                                                       void* kv_buffer, int32_t* lens, int32_t max_len, const void* q,
                                                       const void* k_new, const void* v_new, void* out,
                                                       void* stream) {
  return noalloc_step(cfg, head_labels, kv_buffer, lens, max_len, q, k_new, v_new, out, stream, 0);
}

extern "C" aoh_status aoh_decode_step_noalloc_status(uint32_t* flags, void* stream) {
  if (flags) *flags = 0u;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc_status: cudaStreamSynchronize failed");
  // read and clear the sticky word of the current device's array (no
  // allocation: symbol copies into and out of a host variable)
  uint32_t w = 0u;
  const size_t at = kStatusWord * sizeof(uint32_t);
  e = cudaMemcpyFromSymbol(&w, g_noalloc_scratch, sizeof(w), at, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc_status: cudaMemcpyFromSymbol failed");
  if (w == 0u) return AOH_OK;
  const uint32_t zero = 0u;
  e = cudaMemcpyToSymbol(g_noalloc_scratch, &zero, sizeof(zero), at, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return set_err(AOH_ERR_CUDA, "aoh_decode_step_noalloc_status: cudaMemcpyToSymbol failed");
  if (flags) *flags = w;
  if (w & kErrTimeout)
    return set_err(AOH_ERR_TIMEOUT, "aoh_decode_step_noalloc: a kernel's bounded wait ran out since the last query");
  return set_err(AOH_ERR_CAPACITY,
                 "aoh_decode_step_noalloc: a step found a sequence already holding max_seq tokens since the last query");
}
