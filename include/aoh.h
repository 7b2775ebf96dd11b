/*
 * aoh.h - C ABI of the AoH head-heterogeneous causal attention library
 * (GB300 / sm_103a).
 *
 * The paper (Sec. 5, "Deploying LLMs With AoH") splits the KV heads of every
 * layer into two kinds:
 *   retrieval heads keep the full K/V history and run full causal attention;
 *   streaming heads keep S sink tokens plus the W most recent tokens (a fixed
 *   per-head cache) and attend only to those ("Chunked-Prefill Stage").
 * Query heads inherit the label of their KV head (Appendix "GQA Extension").
 * Each head is computed independently and the outputs sit at their own head
 * index, which is the concatenation of Eq. 8 (the W_O projection that follows
 * is outside this library).
 *
 * Conventions for every call
 *   - Element type of q, k, v, out and of the cache is bfloat16 (2 bytes),
 *     passed as untyped pointers. Accumulation is fp32.
 *   - All tensors are dense, row-major, and live in device memory of the
 *     current CUDA device, unless a parameter says otherwise. Each device
 *     pointer must be 16-byte aligned.
 *   - Query head h belongs to KV head h / (n_q_heads / n_kv_heads).
 *   - A key at position j is visible to the query at position i iff j <= i
 *     and, for a streaming KV head, (j < S or i - j < W): the window counts
 *     the query's own position (aoh_config.chunk = 0, and every decode step).
 *     With aoh_config.chunk = K > 0, prefill rows of a streaming head use
 *     the chunk-eviction rule documented at that field.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream). Calls are asynchronous and stream-ordered; calls that use one
 *     cache must be ordered on one stream (or synchronised by the caller).
 *   - Every call returns a status and never aborts; on failure
 *     aoh_last_error() returns a message for the calling thread. Invalid
 *     arguments are caught on the host before anything is launched.
 *
 * Ownership: the caller allocates and frees the KV buffer, the inputs and the
 * outputs. The handle owns only host state and device arrays it allocates
 * itself: a small metadata block (sequence lengths, split-KV scratch, an
 * error word) and the prefill work list, both allocated by aoh_cache_init,
 * and the H2Share anchor workspace, allocated by aoh_cache_reserve or on the
 * first anchor step; aoh_cache_destroy releases all of it.
 */
#ifndef AOH_H_
#define AOH_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum aoh_status {
  AOH_OK = 0,
  AOH_ERR_INVALID = 1,     /* null pointer, bad shape, misaligned pointer, bad label */
  AOH_ERR_CAPACITY = 2,    /* buffer too small, or a sequence would pass max_seq   */
  AOH_ERR_CUDA = 3,        /* a CUDA runtime call failed                           */
  AOH_ERR_TIMEOUT = 4,     /* a kernel's bounded wait ran out (see aoh_cache_check) */
  AOH_ERR_UNSUPPORTED = 5, /* d_head or group size outside the compiled kernels    */
  AOH_ERR_STATE = 6        /* reserved: call not valid in the cache's current state */
} aoh_status;

/* Labels of a KV head (one uint8 per KV head). */
#define AOH_RETRIEVAL 0
#define AOH_STREAMING 1

typedef struct aoh_config {
  int32_t batch;      /* B: sequences in the cache, >= 1                           */
  int32_t n_q_heads;  /* Hq, a multiple of n_kv_heads                             */
  int32_t n_kv_heads; /* Hkv                                                      */
  int32_t d_head;     /* 64 or 128; n_q_heads / n_kv_heads must be 1-8 or 16 for
                         128, and 1, 2, 4, 7 or 8 for 64 (else UNSUPPORTED)     */
  int32_t max_seq;    /* tokens a retrieval head can hold per sequence, >= 1      */
  int32_t sink;       /* S >= 0: sink tokens kept by a streaming head             */
  int32_t window;     /* W >= 1: recent tokens kept by a streaming head           */
  int32_t chunk;      /* streaming prefill rule: 0 = per-token window (below);
                         K >= 1 = eviction after each K-token chunk (Sec. 5,
                         "Chunked-Prefill Stage"): a prefill row at position i
                         of chunk c = i / K sees keys j <= i with j < S or
                         j >= c*K - W. Decode always uses the per-token rule. */
} aoh_config;

typedef struct aoh_cache aoh_cache; /* opaque handle */

/*
 * Exact byte size of the KV buffer for `cfg` and `head_labels` [n_kv_heads]:
 *   B * (n_R * max_seq + n_S * (S + W)) * d_head * 2 (K and V) * 2 (bf16),
 * n_R / n_S = number of retrieval / streaming KV heads. This is the per-layer
 * KV memory the paper accounts (Appendix "Details on Baseline Budgets" 32K
 * KV-memory table; memory columns of Appendix "Additional Efficiency
 * Results"). Returns 0 if the arguments are invalid (message in
 * aoh_last_error()). Host only.
 */
size_t aoh_cache_bytes(const aoh_config* cfg, const uint8_t* head_labels);

/*
 * Bind a caller-owned device buffer as an empty KV cache (all lengths 0).
 *   cfg          shape and streaming parameters (copied).
 *   head_labels  host array [n_kv_heads] of AOH_RETRIEVAL / AOH_STREAMING
 *                (copied).
 *   kv_buffer    device pointer, 256-byte aligned, at least
 *                aoh_cache_bytes(cfg, head_labels) bytes; its contents need
 *                not be initialised. Not freed by the library.
 *   out          receives the handle.
 * Layout of kv_buffer: first one region per (sequence b, retrieval head) in
 * order b-major, retrieval heads in increasing KV-head index; then one region
 * per (b, streaming head) in the same order. A region is K[capacity][d_head]
 * followed by V[capacity][d_head], capacity = max_seq (retrieval) or S + W
 * (streaming). A retrieval head stores position p at row p. A streaming head
 * stores position p < S at row p and position p >= S at row
 * S + (p - S) mod W (a ring of W rows after the sinks). aoh_cache_region()
 * returns the offsets.
 * Allocates the handle's metadata block and a prefill work list sized for
 * chunks of up to max_seq tokens (B * n_q_heads * ceil(max_seq / 256)
 * entries of 16 bytes), and synchronises the device once (metadata upload).
 * Errors: INVALID, CAPACITY, UNSUPPORTED, CUDA.
 */
aoh_status aoh_cache_init(const aoh_config* cfg, const uint8_t* head_labels, void* kv_buffer,
                          size_t kv_buffer_bytes, aoh_cache** out);

/*
 * Causal prefill of one chunk of every sequence (Sec. 5, "Chunked-Prefill
 * Stage"; every streaming query uses the per-token sink + window rule above).
 * The chunk of sequence b holds positions L_b .. L_b + len_b - 1, where L_b
 * is the number of tokens the cache already holds (0 for a first prefill):
 * its rows attend to the cached prefix (retrieval heads: every earlier
 * position; streaming heads: the sinks and the window, read from the sink and
 * ring slots) and to the chunk itself. Its K/V are then appended (retrieval
 * rows; streaming sinks and the last W positions of the new length).
 *   q    [B][T][n_q_heads][d_head]
 *   k, v [B][T][n_kv_heads][d_head]
 *   T    padded chunk length, >= 1.
 * With aoh_config.chunk = K > 0, every L_b must be a multiple of K (a call
 * starts on a chunk boundary; INVALID otherwise); a call may span several
 * chunks.
 *   seq_lens  host array [B] of chunk lengths 1..T, or NULL (all T). Rows at
 *             or past seq_lens[b] are ignored: their contents (even NaN) do
 *             not affect any output, and their outputs are not written.
 *   out  [B][T][n_q_heads][d_head], or NULL to only fill the cache.
 * With out, the host lists the call's query tiles (longest first) and uploads
 * the list to the handle's work list. A chunk of at most max_seq tokens (or
 * of at most the max_tokens given to aoh_cache_reserve) fits the list as
 * allocated; only a longer chunk, which a cache without retrieval heads can
 * take, grows it with cudaMalloc (which synchronises the device).
 * Errors: INVALID, CAPACITY (a retrieval head would pass max_seq; nothing is
 * launched), CUDA.
 */
aoh_status aoh_prefill(const void* q, const void* k, const void* v, int32_t T,
                       const int32_t* seq_lens, aoh_cache* cache, void* out, void* stream);

/*
 * One decode step for every sequence (Sec. 5 "Decode Stage", Eq. 8): the new
 * token of sequence b sits at position t = len(b); its K/V are appended (the
 * streaming ring overwrites the position that leaves the window) and its
 * query attends over positions visible to it; len(b) becomes t + 1.
 *   q            [B][n_q_heads][d_head]
 *   k_new, v_new [B][n_kv_heads][d_head]
 *   out          [B][n_q_heads][d_head]
 * The lengths advance on the device as well as in the handle, so consecutive
 * steps need no host work between them. Errors: INVALID, CAPACITY (a
 * retrieval head would pass max_seq; nothing is launched), CUDA.
 */
aoh_status aoh_decode_step(const void* q, const void* k_new, const void* v_new, aoh_cache* cache,
                           void* out, void* stream);

/*
 * H2Share anchor layer (the paper's H2Share section; GQA extension
 * appendix): an ordinary decode step (as aoh_decode_step) that also selects,
 * for every sequence b and retrieval KV head, the positions a reuse layer of
 * the same block will borrow. The importance of position j is the sum over
 * the group's query heads of their attention probabilities at j (positions
 * 0..t, the new token included); the min(top_k, t + 1) most important
 * positions are kept, ties to the lower position, in increasing order.
 *   top_k    >= 1.
 *   indices  device int32 [B][n_r][top_k] (n_r = retrieval KV heads, in
 *            increasing KV-head index), written on the stream; entries past
 *            min(top_k, t + 1) are -1.
 * Needs d_head 128 (the tensor-core decode). Uses a workspace of about
 * B * n_r * max_seq * (group size) floats in the handle, plus
 * B * n_r * max_seq more when max_seq exceeds 147456; aoh_cache_reserve
 * allocates it up front, else the first anchor step does (a cudaMalloc,
 * which synchronises the device); aoh_cache_destroy frees it.
 * Errors: INVALID, CAPACITY, UNSUPPORTED, CUDA.
 */
aoh_status aoh_decode_step_anchor(const void* q, const void* k_new, const void* v_new, aoh_cache* cache,
                                  void* out, int32_t top_k, int32_t* indices, void* stream);

/*
 * H2Share reuse layer: a decode step whose retrieval heads attend only to
 * their own K/V at positions borrowed from the block's anchor layer (no K/V
 * crosses layers); streaming heads decode as usual, and the new token is
 * appended for every head as in aoh_decode_step.
 *   indices          device int32 [B][n_anchor_groups][top_k] from
 *                    aoh_decode_step_anchor at the same step (the anchor
 *                    layer holds the same sequence lengths).
 *   n_anchor_groups  the anchor layer's retrieval KV heads, 1..64.
 *   top_k            as given to the anchor step.
 *   group_map        host int32 [n_r]: for this layer's i-th retrieval KV
 *                    head, the anchor retrieval head (0..n_anchor_groups-1)
 *                    whose positions it borrows (the paper maps each reuse
 *                    group to its most similar anchor group, Eq. sim).
 * Retrieval head i of sequence b attends to the first min(top_k, t + 1)
 * entries of its list; entries outside [0, t] are clamped into it (the
 * reads stay in bounds, the result is then unspecified). d_head 128 runs on
 * the tensor cores, the borrowed rows copied by extra gather warps (sixteen
 * for groups of up to four query heads, eight above); d_head 64 on the
 * CUDA-core kernel.
 * Errors: INVALID, CAPACITY, UNSUPPORTED, CUDA.
 */
aoh_status aoh_decode_step_reuse(const void* q, const void* k_new, const void* v_new, aoh_cache* cache,
                                 void* out, const int32_t* indices, int32_t n_anchor_groups, int32_t top_k,
                                 const int32_t* group_map, void* stream);

/*
 * H2Share head mapping (the paper's H2Share section, Eq. sim; GQA extension
 * appendix), offline, from the frozen weights of an anchor layer and a reuse
 * layer. sim(h, h') is the normalised Frobenius inner product of the two
 * kernel matrices M = W_K^T W_Q, computed through traces of d_head x d_head
 * products; a group-pair similarity is the mean over the query-head pairs;
 * each reuse retrieval group maps to the anchor retrieval group of highest
 * similarity (ties to the lower index).
 *   w_q_*  device bf16 [n_q_heads][d_head][d_model]; w_k_* [n_kv_heads][...],
 *          laid out as for aoh_classify; 16-byte aligned; d_model a
 *          multiple of 8; d_head 64 or 128.
 *   anchor_labels, reuse_labels  host uint8 [n_kv_heads] (AOH_RETRIEVAL /
 *          AOH_STREAMING), e.g. from aoh_classify.
 *   map_out        host int32 [n_kv_heads]: for each reuse group, the
 *                  anchor group it borrows from; -1 for streaming reuse
 *                  groups (or when the anchor layer has no retrieval group).
 *                  Listing the retrieval entries in increasing reuse-group
 *                  order, converted to anchor retrieval slots, gives the
 *                  group_map of aoh_decode_step_reuse.
 *   group_sim_out  host double [n_kv_heads][n_kv_heads] (anchor-major), or NULL.
 * The d_model contractions run on the tensor cores (bf16 in, fp32
 * accumulate); traces and norms in fp64. Keeps one device workspace per
 * device for the process (allocated with cudaMalloc on the first call that
 * needs more; calls on a device are serialised) and synchronises `stream`.
 * Errors: INVALID, UNSUPPORTED, TIMEOUT, CUDA.
 */
aoh_status aoh_h2share_map(const void* w_q_anchor, const void* w_k_anchor, const void* w_q_reuse,
                           const void* w_k_reuse, int32_t n_q_heads, int32_t n_kv_heads, int32_t d_head,
                           int32_t d_model, const uint8_t* anchor_labels, const uint8_t* reuse_labels,
                           int32_t* map_out, double* group_sim_out, void* stream);

/*
 * Allocate now the device arrays that later calls would otherwise allocate on
 * first use (the paper has no counterpart): the prefill work list for chunks
 * of up to max_tokens tokens (aoh_cache_init already sized it for max_seq),
 * and, if anchor_workspace is nonzero, the H2Share anchor workspace of
 * aoh_decode_step_anchor. A caller that must not allocate while serving calls
 * this once after aoh_cache_init; calls within these limits then allocate
 * nothing. Uses cudaMalloc (which synchronises the device) for what is not
 * yet allocated. Errors: INVALID, UNSUPPORTED (anchor workspace without the
 * d_head 128 tensor-core decode), CUDA.
 */
aoh_status aoh_cache_reserve(aoh_cache* cache, int32_t max_tokens, int32_t anchor_workspace);

/* Copy the host-side lengths (tokens held per sequence) into lens_out [B]. */
aoh_status aoh_cache_lens(const aoh_cache* cache, int32_t* lens_out);

/*
 * Byte offsets (from kv_buffer) of the K and V rows of sequence b, KV head h,
 * and that region's capacity in rows. Host only; for inspection and tests.
 */
aoh_status aoh_cache_region(const aoh_cache* cache, int32_t b, int32_t kv_head, size_t* k_offset,
                            size_t* v_offset, int32_t* capacity);

/* Mark every sequence empty again (host and device lengths), stream-ordered. */
aoh_status aoh_cache_reset(aoh_cache* cache, void* stream);

/*
 * Synchronise `stream` and read the device error word that kernels set when
 * a bounded wait runs out (or when a decode step finds a sequence already
 * holding max_seq tokens, which the host checks prevent on this handle).
 * Returns AOH_OK, AOH_ERR_TIMEOUT or AOH_ERR_CAPACITY (and clears the word),
 * or AOH_ERR_CUDA.
 */
aoh_status aoh_cache_check(aoh_cache* cache, void* stream);

/*
 * Self-test of the bounded waits every kernel uses (the paper has no
 * counterpart): one warp waits on a barrier that nothing arrives at for
 * limit_ns (1 ms .. 2 s), gives up, and records the timeout in the cache's
 * error word, as a kernel whose partner role stalled would. The next
 * aoh_cache_check returns AOH_ERR_TIMEOUT (and clears the word); the cache
 * and the CUDA context stay usable. *elapsed_ns (may be NULL) receives how
 * long the wait lasted. Synchronises `stream`. Errors: INVALID, CUDA.
 */
aoh_status aoh_cache_selftest_wait(aoh_cache* cache, int64_t limit_ns, int64_t* elapsed_ns, void* stream);

/* Release the handle and its device metadata (not the KV buffer). NULL is a no-op. */
void aoh_cache_destroy(aoh_cache* cache);

/* Message of the last failed call on this thread ("" if none). */
const char* aoh_last_error(void);

/*
 * A decode step for callers that cannot allocate device memory (the paper has
 * no counterpart; this is a deployment convenience of the library).
 *
 * Who needs it: a caller that must not allocate device memory once it is
 * running, e.g. an inference server that reserves its whole memory arena at
 * start-up and treats any later cudaMalloc as an error, or a latency-critical
 * loop that cannot absorb cudaMalloc's implicit device-wide synchronisation.
 * aoh_cache_init allocates a small metadata block, so such callers cannot use
 * the handle API for decode. This call runs the same split-KV decode kernel
 * as aoh_decode_step with no handle and performs no device allocation: its
 * scratch (split partials, arrival counters, an error word) lives in one
 * statically allocated device array of 16 MiB + 128 KiB inside the library,
 * which every GPU that loads the library holds until the process exits.
 *
 *   cfg, head_labels  as for aoh_cache_init (host memory, not retained).
 *   kv_buffer  the KV cache in the layout aoh_cache_init documents (e.g.
 *              filled by aoh_prefill through a handle, or written by the
 *              caller); 256-byte aligned. The new token's K/V is appended.
 *   lens       device int32 [B]: tokens held per sequence before the step;
 *              each entry is advanced by one on the device.
 *   max_len    host upper bound of every lens[b]; used for the split schedule
 *              and the host capacity check (max_len + 1 <= max_seq when a
 *              retrieval head exists). A bound that is too low (e.g. a
 *              CUDA graph captured once and replayed for many steps) still
 *              gives correct outputs, with a less even split.
 *   q, k_new, v_new, out  as for aoh_decode_step.
 *
 * Limits and behaviour:
 *   - batch * n_kv_heads must be <= 16320 (AOH_ERR_CAPACITY otherwise). When
 *     the partial space is too small for the usual split count, fewer splits
 *     are used.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current) and caches it; make
 *     that first call before any stream capture.
 *   - Every call shares the one array. Each call is a single kernel launch,
 *     which leaves the counters that must start at zero at zero when it
 *     ends. Calls whose kernels overlap on the GPU (on different streams, or
 *     from different threads without ordering) race on the scratch and
 *     produce wrong results: order them on one stream.
 *   - The kernel also checks capacity on the device: a sequence whose
 *     lens[b] already equals max_seq (with a retrieval head present) is
 *     skipped: nothing is appended, its outputs are not written and lens[b]
 *     stays as it is. Such a step, and a bounded-wait timeout inside the
 *     kernel (whose outputs are then unspecified), are not reported by this
 *     asynchronous call; they set bits of a sticky status word that
 *     aoh_decode_step_noalloc_status() reads. Either way the launch leaves
 *     the scratch clean for the next call.
 * Errors: INVALID, CAPACITY, UNSUPPORTED, CUDA.
 */
aoh_status aoh_decode_step_noalloc(const aoh_config* cfg, const uint8_t* head_labels, void* kv_buffer,
                                   int32_t* lens, int32_t max_len, const void* q, const void* k_new,
                                   const void* v_new, void* out, void* stream);

/*
 * Status of the allocation-free decode steps on the current device since the
 * last query (the paper has no counterpart). Synchronises `stream` (order
 * every aoh_decode_step_noalloc call of the device on it, or synchronise
 * them first), reads the sticky status word kept in the same static array
 * and clears it; allocates nothing.
 *   flags  host uint32 (may be NULL): 1 = a bounded wait ran out (those
 *          outputs are unspecified), 2 = a step found a sequence already
 *          holding max_seq tokens (that sequence was skipped); 0 if neither.
 * Returns AOH_OK, AOH_ERR_TIMEOUT (bit 1 set), AOH_ERR_CAPACITY (bit 2
 * alone) or AOH_ERR_CUDA.
 */
aoh_status aoh_decode_step_noalloc_status(uint32_t* flags, void* stream);

/*
 * Self-test of the allocation-free step's recovery from a bounded-wait
 * timeout (the paper has no counterpart): the same call and arguments as
 * aoh_decode_step_noalloc, except that in the launch's last CTA (which
 * always holds rows of the step) the softmax warps withhold their first
 * result, so the MMA warp's wait for it runs out (after about 2 s) and that
 * CTA stops once its copies and MMAs in flight have landed; the other CTAs
 * finish. The outputs of this call are unspecified, the new token may be
 * missing from the cache rows that the stalled CTA would have appended,
 * and the lengths advance as usual. The launch still leaves the static scratch clean, and
 * aoh_decode_step_noalloc_status() then reports AOH_ERR_TIMEOUT once.
 * Needs d_head 128 (UNSUPPORTED otherwise). Errors: as
 * aoh_decode_step_noalloc.
 */
aoh_status aoh_decode_step_noalloc_selftest(const aoh_config* cfg, const uint8_t* head_labels, void* kv_buffer,
                                            int32_t* lens, int32_t max_len, const void* q, const void* k_new,
                                            const void* v_new, void* out, void* stream);

/*
 * Effective-rank head classification (Sec. 4, Eq. 2-6 and Algorithm 1;
 * Appendix "GQA Extension"), computed on the GPU in fp64, for n_layers
 * layers at once. For query head h of a layer, M_h = W_K^T W_Q (Eq. 2, the
 * key projection of h's group); its nonzero singular values give
 * ER(h) = exp(entropy of sigma / sum(sigma)) (Eq. 4). A group's score is the
 * mean ER of its query heads; in every layer the
 * ceil((100 - sparsity_pct) * n_kv_heads / 100) lowest groups are labelled
 * retrieval (ties to the lower group index), the rest streaming.
 *   w_q  device bf16 [n_layers][n_q_heads][d_head][d_model]: per layer,
 *        W_Q^h is rows h*d_head .. h*d_head + d_head - 1 of a q_proj weight
 *        stored [n_q_heads * d_head][d_model] (out x in, row-major).
 *   w_k  device bf16 [n_layers][n_kv_heads][d_head][d_model], likewise.
 *   d_head 64 or 128; d_model >= 1; sparsity_pct in [0, 100];
 *   n_layers * (n_q_heads + n_kv_heads) <= 65535.
 *   er_out     host double [n_layers][n_q_heads] receiving ER, or NULL.
 *   labels_out host uint8 [n_layers][n_kv_heads] receiving AOH_RETRIEVAL /
 *              AOH_STREAMING, ready for aoh_cache_init.
 * Work: the Gram matrices W W^T (exact bf16 products, fp64 sums), their
 * semi-definite Cholesky factors L, and a one-sided Jacobi SVD of
 * L_K^T L_Q, whose singular values are those of M_h; singular values at or
 * below sigma_max * d_model * eps are dropped as zeros.
 * Allocates temporary device memory stream-ordered (cudaMallocAsync;
 * about 0.26 MB per matrix at d_head 128), frees it, and synchronises
 * `stream` before returning. Errors: INVALID, UNSUPPORTED, CUDA.
 */
aoh_status aoh_classify(const void* w_q, const void* w_k, int32_t n_layers, int32_t n_q_heads,
                        int32_t n_kv_heads, int32_t d_head, int32_t d_model, int32_t sparsity_pct,
                        double* er_out, uint8_t* labels_out, void* stream);

/* Library ABI version (major * 100 + minor); 101 added aoh_config.chunk, 102
 * aoh_cache_reserve and aoh_decode_step_noalloc_status. */
int32_t aoh_version(void);

#ifdef __cplusplus
}
#endif

#endif /* AOH_H_ */
