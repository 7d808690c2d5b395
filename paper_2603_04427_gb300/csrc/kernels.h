// Internal launch interface between the C ABI (tk_api.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace tk {

// Launch with programmatic stream serialization: the kernel's CTAs may start
// (and run their prologue up to pdl_wait()) while the previous kernel on the
// stream finishes.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

struct DecodeParams {
  const void* q;             // bf16 [B][Hq][R]
  const void* k;             // bf16 or int8 cache / pool
  const void* v;             // bf16 cache / pool
  const float* k_scale;      // fp32 per-token key scales (int8 keys)
  const int32_t* page_table; // [B][max_pages] (paged)
  const int32_t* seq_lens;   // [B]
  void* out;                 // [B][Hq][DV]
  int out_f32;
  float* part;         // [n_cta][2][record] partial (o, m, l) of pairs that straddle CTAs
  int32_t* counters;   // [B][Hkv] arrival counters, zero between launches
  int* err;            // device error word
  int B, Hq, Hkv, R, DV, G;
  int k_fmt;           // key format: 0 bf16, 1 int8, 2 int4 (two codes per byte)
  int capacity;        // contiguous
  int page_size, page_shift, num_pages, max_pages;  // paged (page_size 0 = contiguous)
  int max_seq_len;
  int n_cta;           // grid size (one persistent CTA per SM)
  float scale_log2;    // scale * log2(e)
  // append fused into the decode: seq_lens are the lengths before the append,
  // the new token of (b, g) (k_new [B][Hkv][R], v_new [B][Hkv][DV]) is
  // written at position seq_lens[b] and attended to with the cached ones
  int fuse_append;
  const void* k_new;
  const void* v_new;
};

// Launch plan shared by tk_decode_workspace_size and tk_attn_decode.
struct DecodePlan {
  int n_cta;
  size_t off_counters, off_part, bytes;
};
DecodePlan plan_decode(int B, int Hq, int Hkv, int R, int DV, int k_fmt, int num_sms);
int decode_max_batch();

cudaError_t launch_decode(const DecodeParams& p, cudaStream_t stream, int* unsupported);

struct AppendParams {
  void* k;                   // cache / pool (bf16 or int8 codes)
  void* v;
  float* k_scale;
  const int32_t* page_table;
  const int32_t* seq_lens;
  const void* k_new;         // bf16 [B][Hkv][T][R]
  const void* v_new;         // bf16 [B][Hkv][T][DV]
  int* err;
  int B, Hkv, R, DV, T;
  int k_fmt;   // 0 bf16, 1 int8, 2 int4
  int capacity;
  int page_size, page_shift, num_pages, max_pages;
};

cudaError_t launch_append(const AppendParams& p, cudaStream_t stream, int* unsupported);

struct PrefillParams {
  const void* q;  // bf16 [B][Hq][S][R]
  const void* k;  // bf16 [B][Hkv][S][R], or the cache / pool (cached mode)
  const void* v;  // bf16 [B][Hkv][S][DV], or the cache / pool (cached mode)
  void* out;      // [B][Hq][S][DV]
  int out_f32;
  int* err;
  int B, Hq, Hkv, S, R, DV;
  int causal;
  float scale_log2;
  int num_sms;
  int head_group;  // (b, h) pairs per L2 group, set by the launcher
  // cached mode (a chunk of S queries after seq_lens[b] cached tokens):
  // query i of sequence b sits at position seq_lens[b] + i and the keys are
  // the cache's first seq_lens[b] + S tokens (bottom-right causal)
  const int32_t* seq_lens;  // nullptr: plain prefill (no cache)
  const int32_t* page_table;
  int capacity;             // contiguous cache rows per (b, g)
  int page_size, page_shift, num_pages, max_pages;  // paged (page_size 0 = contiguous)
  int kv_limit;             // bound of seq_lens[b] + S
  int k_fmt;                // cache keys: 0 bf16, 1 int8, 2 int4 (cached mode only)
  const float* k_scale;     // fp32 per-token key scales (int8 / int4 keys)
  float* lse;               // optional [B][Hq][S]: natural-log logsumexp of each row's scores
  // int8 / int4 keys: device workspace the context's keys are widened into
  // (prefill_workspace_bytes(B, Hkv, R, DV, k_fmt, kw_rows) bytes, 256-byte
  // aligned), kw_rows >= kv_limit rows per (b, kv head), a multiple of 4
  void* kw;
  size_t kw_bytes;
  int kw_rows;
  const float* kw_scale;    // set by the launcher: the workspace's scale plane, if any
};

struct BackwardParams {
  const void* q;      // bf16 [B][Hq][S][R]
  const void* k;      // bf16 [B][Hkv][S][R]
  const void* v;      // bf16 [B][Hkv][S][DV]
  const void* out;    // bf16 [B][Hq][S][DV]  forward output
  const void* d_out;  // bf16 [B][Hq][S][DV]  gradient of the loss w.r.t. out
  const float* lse;   // [B][Hq][S] natural-log logsumexp from the forward
  float* dq;          // fp32 [B][Hq][S][R]  (accumulated: zeroed by the preprocessing kernel)
  float* dk;          // fp32 [B][Hkv][S][R]
  float* dv;          // fp32 [B][Hkv][S][DV]
  // workspace, rows padded to S_pad (a multiple of 128) per (b, query head),
  // both negated so that the kernels add them:
  float* nl2;         // [B*Hq][S_pad] -lse * log2(e); -inf on rows >= S (weight 0)
  float* nd;          // [B*Hq][S_pad] -rowsum(d_out * out); 0 on rows >= S
  int* err;
  int B, Hq, Hkv, S, S_pad, R, DV;
  int causal;
  float scale;
};

// Rows of the backward's per-row statistics: S rounded up to 128.
inline int backward_rows(int S) { return (S + 127) / 128 * 128; }

cudaError_t launch_backward(const BackwardParams& p, cudaStream_t stream, int* unsupported);
// The tensor-memory gradient kernel, after the preprocessing pass.
cudaError_t launch_backward_tc(const BackwardParams& p, cudaStream_t stream, int* unsupported);

// Bytes of workspace the prefill of a quantised-key cache needs (0 for bf16
// keys or an unsupported shape).
size_t prefill_workspace_bytes(int B, int Hkv, int R, int DV, int k_fmt, int rows);
cudaError_t launch_prefill(const PrefillParams& p, cudaStream_t stream, int* unsupported);

// One thread waits limit_ns on an mbarrier that nothing arrives at, through the
// library's bounded wait, which records a timeout in *err and returns.
cudaError_t launch_wait_timeout(int* err, uint64_t limit_ns, cudaStream_t stream);

}  // namespace tk
