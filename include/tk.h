/*
 * tk.h -- C ABI of the thin-key ("factored-key") attention library for
 * GB300 (sm_103a).
 *
 * The method (arxiv 2603.04427, "Thin Keys, Full Values"):
 *   Section 2.1, Eqs. 1-4: per head, out = softmax(Q K^T * scale) V where
 *   queries and keys are r wide (the selection dimension d_select/h) and
 *   values keep the full head width d_v.  The paper's scale is
 *   1/sqrt(r) (Eq. 4); it is an explicit argument here.
 *   Section 2.3 (thin-key and absorbed-query equations): only the r-wide
 *   keys are cached; queries arrive already projected to r.
 *   Section 2.4, Eqs. 8-9: the cache holds r + d_v values per token and
 *   kv head.
 *   Section 3.4 / 3.5: thin keys compose with GQA; query head h reads kv
 *   head h / (h_q / h_kv).
 *   Section 6 ("Flash Attention and composability"): thin keys compose
 *   with key quantisation; here int8 keys with one fp32 absmax scale per
 *   token and kv head.
 *
 * Conventions for every entry point:
 *   - Device pointers are raw CUDA device addresses on the current device.
 *     The caller owns every buffer; the library allocates no device memory.
 *   - All work is enqueued on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream) and is asynchronous: no call synchronises, except
 *     tk_get_device_error.
 *   - Argument errors are detected on the host and returned before anything
 *     is launched.  Launch failures return TK_ERR_CUDA.  Bad values that
 *     only the device sees (a page id out of range, a seq_len beyond the
 *     capacity) are clamped to a safe value, recorded in a device error
 *     word and reported by tk_get_device_error; the output is then
 *     unspecified but no access leaves the caller's buffers.
 *   - tk_last_error() returns a human-readable reason for the last non-OK
 *     status returned on the calling host thread.
 *   - Tensors are dense, row-major, innermost dimension last, with base
 *     addresses aligned to 16 bytes.
 *
 * Cache layouts (owned by the caller, described by tk_cache_desc):
 *   contiguous (page_size == 0):
 *     k_cache  [batch][h_kv][capacity][r]   bf16, or int8 codes, or
 *              [batch][h_kv][capacity][r/2] bytes of packed int4 codes
 *     k_scale  [batch][h_kv][capacity]      fp32 (int8 / int4 keys only)
 *     v_cache  [batch][h_kv][capacity][d_v] bf16
 *   paged (page_size > 0): pools shared by all sequences
 *     k_cache  [num_pages][h_kv][page_size][r] (r/2 bytes for int4 keys)
 *     k_scale  [num_pages][h_kv][page_size]
 *     v_cache  [num_pages][h_kv][page_size][d_v]
 *     page_table [batch][max_pages_per_seq] int32: logical token t of
 *     sequence b lives in page page_table[b][t / page_size], slot
 *     t % page_size.
 */
#ifndef TK_H_
#define TK_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TK_ABI_VERSION 4

typedef enum tk_status {
  TK_OK = 0,
  TK_ERR_INVALID_ARG = 1, /* null/misaligned pointer, inconsistent sizes        */
  TK_ERR_UNSUPPORTED = 2, /* valid request this build has no kernel for         */
  TK_ERR_WORKSPACE = 3,   /* workspace missing, misaligned or too small         */
  TK_ERR_CUDA = 4,        /* a CUDA runtime / driver call failed                */
  TK_ERR_DEVICE = 5       /* a kernel recorded a bad index or a timed-out wait  */
} tk_status;

typedef enum tk_dtype {
  TK_BF16 = 0, /* bfloat16                                  */
  TK_F32 = 1,  /* IEEE binary32                             */
  TK_I8 = 2,   /* int8 key codes (value = code * k_scale)   */
  TK_I4 = 3    /* int4 key codes, two per byte (element 2j in bits 0-3,
                  2j+1 in bits 4-7, 4-bit two's complement;
                  value = code * k_scale)                   */
} tk_dtype;

/* Shape of a thin-key / full-value cache.
 *   batch, h_q, h_kv : sequences, query heads, kv heads (h_q % h_kv == 0,
 *                      h_q / h_kv in {1, 2, 4, 8})
 *   r                : thin key width per head, in {16, 32, 64, 128}
 *   d_v              : value width per head, in {64, 128}
 *   capacity         : contiguous only: token slots per (sequence, kv head),
 *                      a positive multiple of 16
 *   page_size        : 0 for contiguous, else tokens per page in
 *                      {16, 32, 64, 128, 256}
 *   num_pages        : paged only: pages in each pool
 *   max_pages_per_seq: paged only: columns of the page table
 *   k_dtype          : TK_BF16, TK_I8 or TK_I4 (TK_I4 needs r >= 32)          */
typedef struct tk_cache_desc {
  int32_t batch;
  int32_t h_q;
  int32_t h_kv;
  int32_t r;
  int32_t d_v;
  int32_t capacity;
  int32_t page_size;
  int32_t num_pages;
  int32_t max_pages_per_seq;
  int32_t k_dtype;
} tk_cache_desc;

/* Append n_new tokens to every sequence of the cache (Section 2.3: the
 * thin keys k' = x W_K' are what the cache stores; Section 2.4: each token
 * adds r + d_v values per kv head).
 *   k_new    : device bf16 [batch][h_kv][n_new][r]    new thin keys
 *   v_new    : device bf16 [batch][h_kv][n_new][d_v]  new values
 *   seq_lens : device int32 [batch], tokens already cached per sequence;
 *              token t of the new block goes to position seq_lens[b] + t.
 *              Not modified: the caller advances it (e.g. += n_new on the
 *              same stream) before the next call.
 *   k_scale  : device fp32 per-token scales (int8 / int4 keys only, else NULL).
 *   page_table: device int32 [batch][max_pages_per_seq] (paged only, else NULL).
 * int8 keys are quantised per (token, kv head): amax = max|k|,
 * scale = amax / 127 (binary32 division, round to nearest), code =
 * clamp(rint(k / scale), -127, 127) (binary32 division, ties to even);
 * amax == 0 stores scale 0 and zero codes.  int4 keys (Section 6's 4-bit
 * composition) use the same scheme with 7 in place of 127 (codes in
 * [-7, 7]), stored two per byte as described at TK_I4.
 * n_new == 0 is a no-op.  Positions beyond the capacity (contiguous) or
 * beyond max_pages_per_seq * page_size (paged) are not written and set the
 * device error word.  Launched with programmatic dependent launch (see
 * tk_attn_decode).                                                          */
tk_status tk_kv_append(const tk_cache_desc* desc, void* k_cache, void* v_cache, float* k_scale,
                       const int32_t* page_table, const int32_t* seq_lens, const void* k_new,
                       const void* v_new, int32_t n_new, void* stream);

/* Causal (or full) prefill attention over one prompt per sequence
 * (Section 2.1, Eqs. 1-4; prefill is the compute-bound case of Appendix E).
 *   q   : device bf16 [batch][h_q][seq][r]
 *   k   : device bf16 [batch][h_kv][seq][r]
 *   v   : device bf16 [batch][h_kv][seq][d_v]
 *   out : device [batch][h_q][seq][d_v], bf16 (out_dtype TK_BF16, round to
 *         nearest even) or fp32 (TK_F32)
 *   scale: multiplies q.k (the paper uses 1/sqrt(r)); must be > 0
 *   causal: nonzero = query i attends to keys 0..i (top-left aligned);
 *           zero = every query attends to all seq keys.
 * Shapes: r in {16, 32, 64, 128}, d_v in {64, 128}, h_q % h_kv == 0,
 * seq >= 0 (seq == 0 is a no-op).  Scores and the weighted sum accumulate
 * in fp32 on the tensor cores; the softmax weights enter the second
 * product rounded to bf16.                                                  */
tk_status tk_attn_prefill(const void* q, const void* k, const void* v, void* out,
                          int32_t out_dtype, int32_t batch, int32_t h_q, int32_t h_kv,
                          int32_t seq, int32_t r, int32_t d_v, float scale, int32_t causal,
                          void* stream);

/* tk_attn_prefill that also writes, for the backward pass, each query row's
 * natural-log logsumexp of its scaled (masked) scores,
 * lse[b][h][i] = ln sum_j exp(scale q_i . k_j)   (float [batch][h_q][seq]).
 * Other arguments, layouts and errors as tk_attn_prefill.                  */
tk_status tk_attn_forward(const void* q, const void* k, const void* v, void* out, float* lse,
                          int32_t out_dtype, int32_t batch, int32_t h_q, int32_t h_kv,
                          int32_t seq, int32_t r, int32_t d_v, float scale, int32_t causal,
                          void* stream);

/* Bytes of workspace tk_attn_backward needs: two floats per query row (each
 * row's -lse log2 e and -rowsum(d_out * out)), rows padded to a multiple of
 * 128 per (sequence, query head); 0 for invalid arguments.                  */
size_t tk_backward_workspace_size(int32_t batch, int32_t h_q, int32_t seq);

/* Gradients of prefill attention (the training path of thin-key attention;
 * Section 2.1, Eqs. 1-4 differentiated).  For a loss with dL/d(out) = d_out:
 *   dq = scale dS k,  dk = scale dS^T q,  dv = P^T d_out,
 *   dS = P * (d_out v^T - D),  D_i = sum_c d_out_ic out_ic,  P = softmax rows,
 * with a kv head's dk and dv summed over its h_q / h_kv query heads.
 *   q, k, v : the forward's inputs (bf16, layouts of tk_attn_prefill)
 *   out     : the forward's output, bf16 [batch][h_q][seq][d_v]
 *   d_out   : bf16 [batch][h_q][seq][d_v]
 *   lse     : the forward's row logsumexp (tk_attn_forward)
 *   dq      : float [batch][h_q][seq][r]    (overwritten)
 *   dk      : float [batch][h_kv][seq][r]   (overwritten)
 *   dv      : float [batch][h_kv][seq][d_v] (overwritten)
 *   workspace: tk_backward_workspace_size bytes, 256-byte aligned (scratch)
 *   scale, causal: as in the forward.
 * The products run on the tensor cores with bf16 operands (P and dS rounded
 * to bf16) and fp32 accumulation (tcgen05, accumulators in tensor memory);
 * dq is accumulated across key tiles with fp32 reduce-adds, so its
 * low bits may vary run to run.  Two launches (preprocessing, gradients).    */
tk_status tk_attn_backward(const void* q, const void* k, const void* v, const void* out,
                           const void* d_out, const float* lse, float* dq, float* dk, float* dv,
                           void* workspace, size_t workspace_bytes, int32_t batch, int32_t h_q,
                           int32_t h_kv, int32_t seq, int32_t r, int32_t d_v, float scale,
                           int32_t causal, void* stream);

/* Prefill of a chunk of `seq` new tokens per sequence against the cache
 * (Section 2.1, Eqs. 1-4, over a context that continues an existing one):
 * first writes the chunk's thin keys and values at positions
 * seq_lens[b] .. seq_lens[b] + seq - 1 exactly as tk_kv_append (int8 / int4
 * keys quantised the same way, bit for bit), then computes, for query i of
 * the chunk (position seq_lens[b] + i), attention over the cache's tokens
 * 0 .. seq_lens[b] + i (causal, aligned to the end of the context) or over
 * all seq_lens[b] + seq of them (causal == 0).
 *   q        : device bf16 [batch][h_q][seq][r]       the chunk's queries
 *   k_scale  : device fp32 per-token key scales (int8 / int4 keys, else NULL)
 *   k_new    : device bf16 [batch][h_kv][seq][r]      the chunk's thin keys
 *   v_new    : device bf16 [batch][h_kv][seq][d_v]    the chunk's values
 *   seq_lens : device int32 [batch], tokens cached before the chunk (not
 *              modified; the caller advances it by seq afterwards)
 *   max_seq_len: host bound of seq_lens[b] + seq
 *   out      : device [batch][h_q][seq][d_v], TK_BF16 or TK_F32
 *   workspace: int8 / int4 keys: device scratch of
 *              tk_prefill_cached_workspace_size(desc, max_seq_len) bytes,
 *              256-byte aligned (else TK_ERR_WORKSPACE); unused (may be
 *              NULL) for bf16 keys.  Overwritten by every call; reusable by
 *              later calls in stream order.
 * Keys of every k_dtype (Section 6: thin keys compose with key
 * quantisation): the products run on the tensor cores from bf16 tiles.
 * int8 / int4 keys are first widened, once per token of each context, into
 * the workspace: for r <= 64 each key scale * code becomes two bf16 terms
 * hi + lo (within 2^-17 of it, relative) and S = Q hi^T + Q lo^T; for
 * r = 128 the codes become exact bf16 and each score q . code is multiplied
 * by its key's fp32 scale.  Contiguous or paged caches; a sequence whose
 * chunk does not fit sets the device error word and is computed over a
 * clamped context.  Cache slots past a sequence's context may hold anything
 * (they are never weighted).  seq_lens[b] == 0 gives the plain causal
 * prefill of the chunk.  Launches in stream order: append, (key widening,)
 * attention.                                                              */
tk_status tk_attn_prefill_cached(const tk_cache_desc* desc, const void* q, void* k_cache,
                                 void* v_cache, float* k_scale, const int32_t* page_table,
                                 const int32_t* seq_lens, const void* k_new, const void* v_new,
                                 int32_t seq, int32_t max_seq_len, void* out, int32_t out_dtype,
                                 float scale, int32_t causal, void* workspace,
                                 size_t workspace_bytes, void* stream);

/* Bytes of workspace tk_attn_prefill_cached needs for a cache of this shape
 * and this bound of seq_lens[b] + seq: two bf16 planes of r per token and kv
 * head (r <= 64), or one plane and one fp32 scale per token (r = 128), over
 * min(max_seq_len, the cache's tokens per sequence) rows rounded up to a
 * multiple of 4.  0 for bf16 keys or an invalid descriptor.              */
size_t tk_prefill_cached_workspace_size(const tk_cache_desc* desc, int32_t max_seq_len);

/* Bytes of decode workspace needed for a cache of this shape when no
 * sequence is longer than max_seq_len, on the current device (the split of
 * the context depends on its SM count).  0 means the arguments are invalid.
 * The workspace must be zero-filled once before its first use.  It holds
 * per-(sequence, kv head) arrival counters, which every completed
 * tk_attn_decode call leaves at zero again, and split partials, which are
 * scratch; so it can be reused by later calls in stream order (never by two
 * calls that may run concurrently).                                         */
size_t tk_decode_workspace_size(const tk_cache_desc* desc, int32_t max_seq_len);

/* Single-token decode attention over the cache (Section 2.1, Eq. 4 with one
 * query row; the bandwidth-bound case of Section 4.2).
 *   q        : device bf16 [batch][h_q][r], one query token per sequence
 *   seq_lens : device int32 [batch], context length of each sequence
 *              (0 gives a zero output row)
 *   max_seq_len: host upper bound of seq_lens, sizes the launch; a larger
 *              device value is clamped to it and flagged.
 *   out      : [batch][h_q][d_v], TK_F32 or TK_BF16: device memory, or
 *              page-locked host memory (cudaHostAlloc / cudaHostRegister):
 *              under unified addressing the kernel then stores the rows
 *              straight into host memory (zero-copy), which replaces a
 *              separate device-to-host copy when the result is wanted on the
 *              host.  Like every pointer here it is not validated: any other
 *              memory faults like an invalid device pointer.
 *   scale    : multiplies q.k (for int8 keys, q.(code * k_scale))
 *   workspace: device scratch of tk_decode_workspace_size bytes, aligned to
 *              256 bytes (see tk_decode_workspace_size).
 * batch <= 1024 (the kernel keeps per-sequence prefix sums in shared
 * memory); a larger batch returns TK_ERR_UNSUPPORTED.
 * The context is split into fixed token ranges processed in parallel and
 * merged in the same launch; results are deterministic run to run.
 * The kernel is launched with programmatic dependent launch: its CTAs may
 * start while the previous kernel on `stream` finishes, but they touch
 * device memory only after that kernel has completed.                      */
tk_status tk_attn_decode(const tk_cache_desc* desc, const void* q, const void* k_cache,
                         const void* v_cache, const float* k_scale, const int32_t* page_table,
                         const int32_t* seq_lens, int32_t max_seq_len, void* out,
                         int32_t out_dtype, float scale, void* workspace,
                         size_t workspace_bytes, void* stream);

/* One decode step with the append fused in: for every sequence, writes the
 * new token's thin key and value at position seq_lens[b] exactly as
 * tk_kv_append with n_new = 1 (Section 2.3: the cache keeps k' = x W_K';
 * int8 keys quantised the same way, bit for bit), then attends q over the
 * seq_lens[b] + 1 cached tokens exactly as tk_attn_decode with those
 * lengths (Section 2.1, Eq. 4) -- one launch instead of two.
 *   seq_lens : device int32 [batch], tokens cached BEFORE the append (not
 *              modified; the caller advances it by one afterwards)
 *   k_new    : device bf16 [batch][h_kv][r]    the new thin keys
 *   v_new    : device bf16 [batch][h_kv][d_v]  the new values
 *   max_seq_len: host upper bound of seq_lens[b] + 1
 *   The other arguments, the workspace and the errors are those of
 *   tk_attn_decode (k_cache, v_cache and k_scale are written).  A sequence
 *   whose new position does not fit (seq_lens[b] + 1 beyond max_seq_len,
 *   the capacity or the page table) gets no write, is attended over its
 *   clamped length and sets the device error word.  The result equals
 *   tk_kv_append followed by tk_attn_decode bit for bit.                   */
tk_status tk_attn_decode_append(const tk_cache_desc* desc, const void* q, void* k_cache,
                                void* v_cache, float* k_scale, const int32_t* page_table,
                                const int32_t* seq_lens, const void* k_new, const void* v_new,
                                int32_t max_seq_len, void* out, int32_t out_dtype, float scale,
                                void* workspace, size_t workspace_bytes, void* stream);

/* Stream-ordered copy of `bytes` bytes between any two of device memory and
 * page-locked host memory (cudaMemcpyAsync with the direction taken from the
 * pointers), for serving loops that bring a step's inputs from the host:
 * issued natively, it costs the step less host time than a copy through a
 * framework.  bytes == 0 is a no-op; NULL pointers give TK_ERR_INVALID_ARG,
 * a failed enqueue TK_ERR_CUDA.  Not part of the paper's method.            */
tk_status tk_copy_async(void* dst, const void* src, size_t bytes, void* stream);

/* CUDA-graph capture of a serving step, for loops that repeat the same calls
 * on fixed buffers: tk_graph_begin starts capturing `stream` (relaxed mode,
 * so the entry points' host-side set-up may run during the capture); every
 * call enqueued on that stream until tk_graph_end (tk_copy_async, decode,
 * append, prefill) is recorded instead of run; tk_graph_end stops the capture
 * and returns an executable graph in *graph_out.  tk_graph_launch replays it
 * on a stream (one launch for the whole step: far less host time per step
 * than issuing each call); the replay uses the recorded pointers and sizes,
 * so the contents of the buffers (queries, seq_lens, page table, host input
 * buffer) may change between replays but not their addresses.
 * tk_graph_destroy frees the graph.  Errors: NULL stream / graph pointers give
 * TK_ERR_INVALID_ARG; a failed CUDA call gives TK_ERR_CUDA (a capture that
 * fails inside tk_graph_end is ended and discarded).  Not part of the paper's
 * method.                                                                    */
tk_status tk_graph_begin(void* stream);
tk_status tk_graph_end(void* stream, void** graph_out);
tk_status tk_graph_launch(void* graph, void* stream);
tk_status tk_graph_destroy(void* graph);

/* Size of the fixed device scratch array used by tk_attn_decode_noalloc. */
#define TK_DECODE_NOALLOC_SCRATCH_BYTES (8u << 20)

/* tk_attn_decode without a workspace argument, for callers that cannot
 * allocate device memory: runtimes whose device memory is entirely held by
 * their own pool and that forbid cudaMalloc on the decode path (it
 * synchronises the device and can fail), plugin hosts that pass a plugin only
 * its inputs and outputs, and real-time loops that must not touch an
 * allocator between steps.  The paper has no counterpart; this is an
 * interface convenience around the same decode kernel.
 *   Arguments, layouts, results and errors are those of tk_attn_decode.
 *   The split partials and arrival counters live in one static device array
 *   of TK_DECODE_NOALLOC_SCRATCH_BYTES (8 MiB) in this library, which every
 *   GPU that loads the library keeps until the process exits.  A shape whose
 *   tk_decode_workspace_size exceeds it is rejected with TK_ERR_WORKSPACE
 *   (tk_last_error gives both sizes) before anything is launched.
 *   No device memory is allocated or freed.  Every call looks up the
 *   array's device address for the calling thread's current device
 *   (cudaGetSymbolAddress, which allocates nothing; the first lookup on a
 *   device may load the library's device code there, so make the first call
 *   on each device before any stream capture).  A call that passes every
 *   check clears the counters with one cudaMemsetAsync on `stream` just
 *   before its launch; a rejected call writes nothing.
 *   All calls on a device share the array and it keeps the last call's
 *   contents: calls that may overlap on the GPU (different streams without
 *   ordering between them) race and give wrong results.                   */
tk_status tk_attn_decode_noalloc(const tk_cache_desc* desc, const void* q, const void* k_cache,
                                 const void* v_cache, const float* k_scale,
                                 const int32_t* page_table, const int32_t* seq_lens,
                                 int32_t max_seq_len, void* out, int32_t out_dtype, float scale,
                                 void* stream);

/* Synchronise `stream`, then read and clear the device error word of the
 * current device: *code_out = 0 if no kernel recorded an error since the
 * last call, else a nonzero code (1 = index out of range, 2 = a wait timed
 * out).  Returns TK_ERR_DEVICE when the word was nonzero.                  */
tk_status tk_get_device_error(int32_t* code_out, void* stream);

/* Diagnostic of the failure detection (not part of the paper's method).
 * Every wait inside the library's kernels gives up after 1 s, records code 2
 * in the device error word and lets its kernel return instead of spinning.
 * This call exercises that path: it launches one thread that waits, through
 * the same bounded wait, on an mbarrier that nothing ever arrives at, with a
 * limit of limit_us microseconds (1 .. 1000000) in place of the 1 s.  The
 * wait runs out, code 2 is recorded and the kernel returns; the context stays
 * usable.  The next tk_get_device_error returns TK_ERR_DEVICE with
 * *code_out == 2.  A limit outside the range gives TK_ERR_INVALID_ARG.     */
tk_status tk_check_wait_timeout(int32_t limit_us, void* stream);

/* Static string naming a status code.                                      */
const char* tk_status_string(tk_status status);

/* Reason for the last non-OK status returned on this host thread ("" if
 * none).  The pointer stays valid until the next call on this thread.      */
const char* tk_last_error(void);

/* TK_ABI_VERSION of the loaded library.                                     */
int32_t tk_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TK_H_ */
