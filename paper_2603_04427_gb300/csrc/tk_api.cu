// C ABI of the thin-key attention library (declared in include/tk.h):
// argument validation, split planning, the device error word, and dispatch
// to the kernels.  Nothing here allocates device memory.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#include "kernels.h"
#include "tk.h"

namespace {

// Device error word: kernels record the first bad index / timed-out wait here.
__device__ int g_tk_device_error;

constexpr int kMaxDevices = 64;

struct DeviceInfo {
  int num_sms = 0;
  int* err = nullptr;  // device address of g_tk_device_error
};
int g_num_sms[kMaxDevices];  // 0 until read
std::mutex g_dev_mu;

thread_local std::string t_last_error;

tk_status fail(tk_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
tk_status fail(tk_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  t_last_error = buf;
  return s;
}

tk_status cuda_fail(cudaError_t e, const char* what) {
  return fail(TK_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Per-call device facts for the current device: its SM count (read once per
// device and kept) and the device address of the error word.  The address is
// looked up on every call (cudaGetSymbolAddress allocates nothing): after a
// cudaDeviceReset the library's device code is loaded again, possibly at
// another address, and a cached pointer would be stale.
tk_status device_info(DeviceInfo* out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(TK_ERR_UNSUPPORTED, "device ordinal %d", dev);
  {
    std::lock_guard<std::mutex> lock(g_dev_mu);
    if (g_num_sms[dev] == 0) {
      e = cudaDeviceGetAttribute(&g_num_sms[dev], cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) {
        g_num_sms[dev] = 0;
        return cuda_fail(e, "cudaDeviceGetAttribute");
      }
    }
    out->num_sms = g_num_sms[dev];
  }
  e = cudaGetSymbolAddress(reinterpret_cast<void**>(&out->err), g_tk_device_error);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(error word)");
  return TK_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }
int log2i(int x) {
  int s = 0;
  while ((1 << s) < x) ++s;
  return s;
}
bool supported_r(int r) { return r == 16 || r == 32 || r == 64 || r == 128; }
bool supported_dv(int d) { return d == 64 || d == 128; }
bool supported_g(int g) { return g == 1 || g == 2 || g == 4 || g == 8; }

tk_status check_desc(const tk_cache_desc* d) {
  if (!d) return fail(TK_ERR_INVALID_ARG, "desc is NULL");
  if (d->batch < 0 || d->h_q <= 0 || d->h_kv <= 0)
    return fail(TK_ERR_INVALID_ARG, "batch=%d h_q=%d h_kv=%d", d->batch, d->h_q, d->h_kv);
  if (d->h_q % d->h_kv != 0)
    return fail(TK_ERR_INVALID_ARG, "h_q=%d is not a multiple of h_kv=%d", d->h_q, d->h_kv);
  if (!supported_g(d->h_q / d->h_kv))
    return fail(TK_ERR_UNSUPPORTED, "h_q/h_kv=%d (supported: 1, 2, 4, 8)", d->h_q / d->h_kv);
  if (!supported_r(d->r)) return fail(TK_ERR_UNSUPPORTED, "r=%d (supported: 16, 32, 64, 128)", d->r);
  if (!supported_dv(d->d_v)) return fail(TK_ERR_UNSUPPORTED, "d_v=%d (supported: 64, 128)", d->d_v);
  if (d->k_dtype != TK_BF16 && d->k_dtype != TK_I8 && d->k_dtype != TK_I4)
    return fail(TK_ERR_UNSUPPORTED, "k_dtype=%d (supported: TK_BF16, TK_I8, TK_I4)", d->k_dtype);
  if (d->k_dtype == TK_I4 && d->r < 32)
    return fail(TK_ERR_UNSUPPORTED, "r=%d with TK_I4 keys (supported: 32, 64, 128)", d->r);
  if (d->page_size == 0) {
    if (d->capacity <= 0 || d->capacity % 16 != 0)
      return fail(TK_ERR_INVALID_ARG, "capacity=%d must be a positive multiple of 16", d->capacity);
  } else {
    if (!pow2(d->page_size) || d->page_size < 16 || d->page_size > 256)
      return fail(TK_ERR_UNSUPPORTED, "page_size=%d (supported: 16..256, power of two)",
                  d->page_size);
    if (d->num_pages <= 0 || d->max_pages_per_seq <= 0)
      return fail(TK_ERR_INVALID_ARG, "num_pages=%d max_pages_per_seq=%d", d->num_pages,
                  d->max_pages_per_seq);
  }
  return TK_OK;
}

// Key format index used by the kernels: 0 bf16, 1 int8, 2 int4.
int key_format(int32_t k_dtype) { return k_dtype == TK_I8 ? 1 : (k_dtype == TK_I4 ? 2 : 0); }

tk_status check_cache_ptrs(const tk_cache_desc* d, const void* k, const void* v, const void* ks,
                           const void* pt) {
  if (!k || !v) return fail(TK_ERR_INVALID_ARG, "k_cache / v_cache is NULL");
  if (!aligned16(k) || !aligned16(v) || (ks && !aligned16(ks)))
    return fail(TK_ERR_INVALID_ARG, "cache pointers must be 16-byte aligned");
  if ((d->k_dtype == TK_I8 || d->k_dtype == TK_I4) && !ks)
    return fail(TK_ERR_INVALID_ARG, "int8 / int4 keys need k_scale");
  if (d->page_size != 0 && !pt) return fail(TK_ERR_INVALID_ARG, "paged cache needs page_table");
  return TK_OK;
}

}  // namespace

extern "C" {

tk_status tk_kv_append(const tk_cache_desc* desc, void* k_cache, void* v_cache, float* k_scale,
                       const int32_t* page_table, const int32_t* seq_lens, const void* k_new,
                       const void* v_new, int32_t n_new, void* stream) {
  tk_status s = check_desc(desc);
  if (s != TK_OK) return s;
  if (n_new < 0) return fail(TK_ERR_INVALID_ARG, "n_new=%d", n_new);
  if (n_new == 0 || desc->batch == 0) return TK_OK;
  if ((s = check_cache_ptrs(desc, k_cache, v_cache, k_scale, page_table)) != TK_OK) return s;
  if (!seq_lens || !k_new || !v_new) return fail(TK_ERR_INVALID_ARG, "seq_lens / k_new / v_new is NULL");
  if (!aligned16(k_new) || !aligned16(v_new))
    return fail(TK_ERR_INVALID_ARG, "k_new / v_new must be 16-byte aligned");
  DeviceInfo dev;
  if ((s = device_info(&dev)) != TK_OK) return s;
  tk::AppendParams p{};
  p.k = k_cache; p.v = v_cache; p.k_scale = k_scale; p.page_table = page_table;
  p.seq_lens = seq_lens; p.k_new = k_new; p.v_new = v_new; p.err = dev.err;
  p.B = desc->batch; p.Hkv = desc->h_kv; p.R = desc->r; p.DV = desc->d_v; p.T = n_new;
  p.k_fmt = key_format(desc->k_dtype);
  p.capacity = desc->capacity;
  p.page_size = desc->page_size;
  p.page_shift = desc->page_size ? log2i(desc->page_size) : 0;
  p.num_pages = desc->num_pages; p.max_pages = desc->max_pages_per_seq;
  int uns = 0;
  cudaError_t e = tk::launch_append(p, static_cast<cudaStream_t>(stream), &uns);
  if (uns) return fail(TK_ERR_UNSUPPORTED, "append: no kernel for this shape");
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  return TK_OK;
}

namespace {
tk_status prefill_impl(const void* q, const void* k, const void* v, void* out, float* lse,
                       int32_t out_dtype, int32_t batch, int32_t h_q, int32_t h_kv, int32_t seq,
                       int32_t r, int32_t d_v, float scale, int32_t causal, void* stream);
}  // namespace

tk_status tk_attn_prefill(const void* q, const void* k, const void* v, void* out,
                          int32_t out_dtype, int32_t batch, int32_t h_q, int32_t h_kv,
                          int32_t seq, int32_t r, int32_t d_v, float scale, int32_t causal,
                          void* stream) {
  return prefill_impl(q, k, v, out, nullptr, out_dtype, batch, h_q, h_kv, seq, r, d_v, scale,
                      causal, stream);
}

tk_status tk_attn_forward(const void* q, const void* k, const void* v, void* out, float* lse,
                          int32_t out_dtype, int32_t batch, int32_t h_q, int32_t h_kv,
                          int32_t seq, int32_t r, int32_t d_v, float scale, int32_t causal,
                          void* stream) {
  if (seq > 0 && batch > 0 && !lse) return fail(TK_ERR_INVALID_ARG, "lse is NULL");
  return prefill_impl(q, k, v, out, lse, out_dtype, batch, h_q, h_kv, seq, r, d_v, scale,
                      causal, stream);
}

size_t tk_backward_workspace_size(int32_t batch, int32_t h_q, int32_t seq) {
  if (batch < 0 || h_q <= 0 || seq < 0) return 0;
  // two float arrays (-lse log2 e and -rowsum(d_out * out)) of backward_rows(seq) per (b, h)
  return 2 * ((static_cast<size_t>(batch) * h_q * tk::backward_rows(seq) * 4 + 255) / 256 * 256);
}

tk_status tk_attn_backward(const void* q, const void* k, const void* v, const void* out,
                           const void* d_out, const float* lse, float* dq, float* dk, float* dv,
                           void* workspace, size_t workspace_bytes, int32_t batch, int32_t h_q,
                           int32_t h_kv, int32_t seq, int32_t r, int32_t d_v, float scale,
                           int32_t causal, void* stream) {
  if (batch < 0 || seq < 0 || h_q <= 0 || h_kv <= 0)
    return fail(TK_ERR_INVALID_ARG, "batch=%d seq=%d h_q=%d h_kv=%d", batch, seq, h_q, h_kv);
  if (h_q % h_kv != 0) return fail(TK_ERR_INVALID_ARG, "h_q=%d not a multiple of h_kv=%d", h_q, h_kv);
  if (!supported_r(r)) return fail(TK_ERR_UNSUPPORTED, "r=%d (supported: 16, 32, 64, 128)", r);
  if (!supported_dv(d_v)) return fail(TK_ERR_UNSUPPORTED, "d_v=%d (supported: 64, 128)", d_v);
  if (!std::isfinite(scale) || !(scale > 0.f))
    return fail(TK_ERR_INVALID_ARG, "scale must be finite and positive");
  if (batch == 0 || seq == 0) return TK_OK;
  if (!q || !k || !v || !out || !d_out || !lse || !dq || !dk || !dv)
    return fail(TK_ERR_INVALID_ARG, "a tensor pointer is NULL");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || !aligned16(d_out) ||
      !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
    return fail(TK_ERR_INVALID_ARG, "tensors must be 16-byte aligned");
  const size_t need = tk_backward_workspace_size(batch, h_q, seq);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 || workspace_bytes < need)
    return fail(TK_ERR_WORKSPACE, "workspace needs %zu bytes, 256-byte aligned", need);
  DeviceInfo dev;
  tk_status s = device_info(&dev);
  if (s != TK_OK) return s;
  tk::BackwardParams p{};
  p.q = q; p.k = k; p.v = v; p.out = out; p.d_out = d_out; p.lse = lse;
  p.dq = dq; p.dk = dk; p.dv = dv; p.err = dev.err;
  p.S_pad = tk::backward_rows(seq);
  const size_t half = need / 2;   // each array 256-byte aligned
  p.nl2 = static_cast<float*>(workspace);
  p.nd = reinterpret_cast<float*>(static_cast<unsigned char*>(workspace) + half);
  p.B = batch; p.Hq = h_q; p.Hkv = h_kv; p.S = seq; p.R = r; p.DV = d_v;
  p.causal = causal != 0;
  p.scale = scale;
  int uns = 0;
  cudaError_t e = tk::launch_backward(p, static_cast<cudaStream_t>(stream), &uns);
  if (uns) return fail(TK_ERR_UNSUPPORTED, "backward: no kernel for r=%d d_v=%d", r, d_v);
  if (e != cudaSuccess) return cuda_fail(e, "backward launch");
  return TK_OK;
}

namespace {
tk_status prefill_impl(const void* q, const void* k, const void* v, void* out, float* lse,
                       int32_t out_dtype, int32_t batch, int32_t h_q, int32_t h_kv, int32_t seq,
                       int32_t r, int32_t d_v, float scale, int32_t causal, void* stream) {
  if (batch < 0 || seq < 0 || h_q <= 0 || h_kv <= 0)
    return fail(TK_ERR_INVALID_ARG, "batch=%d seq=%d h_q=%d h_kv=%d", batch, seq, h_q, h_kv);
  if (h_q % h_kv != 0) return fail(TK_ERR_INVALID_ARG, "h_q=%d not a multiple of h_kv=%d", h_q, h_kv);
  if (!supported_r(r)) return fail(TK_ERR_UNSUPPORTED, "r=%d (supported: 16, 32, 64, 128)", r);
  if (!supported_dv(d_v)) return fail(TK_ERR_UNSUPPORTED, "d_v=%d (supported: 64, 128)", d_v);
  if (out_dtype != TK_BF16 && out_dtype != TK_F32)
    return fail(TK_ERR_UNSUPPORTED, "out_dtype=%d (supported: TK_BF16, TK_F32)", out_dtype);
  if (!std::isfinite(scale) || !(scale > 0.f))
    return fail(TK_ERR_INVALID_ARG, "prefill scale must be finite and positive");
  if (batch == 0 || seq == 0) return TK_OK;
  if (!q || !k || !v || !out) return fail(TK_ERR_INVALID_ARG, "q / k / v / out is NULL");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out))
    return fail(TK_ERR_INVALID_ARG, "q / k / v / out must be 16-byte aligned");
  DeviceInfo dev;
  tk_status s = device_info(&dev);
  if (s != TK_OK) return s;
  tk::PrefillParams p{};
  p.q = q; p.k = k; p.v = v; p.out = out; p.out_f32 = out_dtype == TK_F32; p.err = dev.err;
  p.B = batch; p.Hq = h_q; p.Hkv = h_kv; p.S = seq; p.R = r; p.DV = d_v;
  p.causal = causal != 0;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.num_sms = dev.num_sms;
  p.lse = lse;
  int uns = 0;
  cudaError_t e = tk::launch_prefill(p, static_cast<cudaStream_t>(stream), &uns);
  if (uns) return fail(TK_ERR_UNSUPPORTED, "prefill: no kernel for r=%d d_v=%d", r, d_v);
  if (e != cudaSuccess) return cuda_fail(e, "prefill launch");
  return TK_OK;
}
}  // namespace

namespace {
// Rows per (b, kv head) of the prefill's widened-key workspace: the bound of
// seq_lens[b] + seq within the cache, rounded up to a multiple of 4.
int prefill_kw_rows(const tk_cache_desc* d, int32_t max_seq_len) {
  const int cache_tokens = d->page_size ? d->max_pages_per_seq * d->page_size : d->capacity;
  return (std::min(max_seq_len, cache_tokens) + 3) / 4 * 4;
}
}  // namespace

tk_status tk_attn_prefill_cached(const tk_cache_desc* desc, const void* q, void* k_cache,
                                 void* v_cache, float* k_scale, const int32_t* page_table,
                                 const int32_t* seq_lens, const void* k_new, const void* v_new,
                                 int32_t seq, int32_t max_seq_len, void* out, int32_t out_dtype,
                                 float scale, int32_t causal, void* workspace,
                                 size_t workspace_bytes, void* stream) {
  tk_status s = check_desc(desc);
  if (s != TK_OK) return s;
  if (seq < 0 || max_seq_len < seq)
    return fail(TK_ERR_INVALID_ARG, "seq=%d max_seq_len=%d", seq, max_seq_len);
  if (out_dtype != TK_BF16 && out_dtype != TK_F32)
    return fail(TK_ERR_UNSUPPORTED, "out_dtype=%d (supported: TK_BF16, TK_F32)", out_dtype);
  if (!std::isfinite(scale) || !(scale > 0.f))
    return fail(TK_ERR_INVALID_ARG, "prefill scale must be finite and positive");
  if (desc->batch == 0 || seq == 0) return TK_OK;
  if ((s = check_cache_ptrs(desc, k_cache, v_cache, k_scale, page_table)) != TK_OK) return s;
  if (!q || !out || !seq_lens || !k_new || !v_new)
    return fail(TK_ERR_INVALID_ARG, "q / out / seq_lens / k_new / v_new is NULL");
  if (!aligned16(q) || !aligned16(out) || !aligned16(k_new) || !aligned16(v_new))
    return fail(TK_ERR_INVALID_ARG, "q / out / k_new / v_new must be 16-byte aligned");
  const int cache_tokens = desc->page_size ? desc->max_pages_per_seq * desc->page_size
                                           : desc->capacity;
  const int kv_limit = std::min(max_seq_len, cache_tokens);
  if (kv_limit < seq)
    return fail(TK_ERR_INVALID_ARG, "seq=%d does not fit the cache (%d tokens)", seq, kv_limit);
  const bool quant = desc->k_dtype != TK_BF16;
  const int kw_rows = quant ? prefill_kw_rows(desc, max_seq_len) : 0;
  if (quant) {
    const size_t need = tk::prefill_workspace_bytes(desc->batch, desc->h_kv, desc->r, desc->d_v,
                                                    key_format(desc->k_dtype), kw_rows);
    if (need == 0)
      return fail(TK_ERR_UNSUPPORTED, "prefill: no kernel for r=%d d_v=%d k_dtype=%d", desc->r,
                  desc->d_v, desc->k_dtype);
    if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 256 != 0)
      return fail(TK_ERR_WORKSPACE, "workspace is NULL or not 256-byte aligned");
    if (workspace_bytes < need)
      return fail(TK_ERR_WORKSPACE, "workspace has %zu bytes, %zu needed", workspace_bytes, need);
  }
  DeviceInfo dev;
  if ((s = device_info(&dev)) != TK_OK) return s;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  // 1. the chunk's keys and values into the cache at seq_lens[b]
  tk::AppendParams a{};
  a.k = k_cache; a.v = v_cache; a.k_scale = quant ? k_scale : nullptr; a.page_table = page_table;
  a.seq_lens = seq_lens; a.k_new = k_new; a.v_new = v_new; a.err = dev.err;
  a.B = desc->batch; a.Hkv = desc->h_kv; a.R = desc->r; a.DV = desc->d_v; a.T = seq;
  a.k_fmt = key_format(desc->k_dtype);
  a.capacity = desc->capacity;
  a.page_size = desc->page_size;
  a.page_shift = desc->page_size ? log2i(desc->page_size) : 0;
  a.num_pages = desc->num_pages; a.max_pages = desc->max_pages_per_seq;
  int uns = 0;
  cudaError_t e = tk::launch_append(a, st, &uns);
  if (uns) return fail(TK_ERR_UNSUPPORTED, "append: no kernel for r=%d d_v=%d", desc->r, desc->d_v);
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  // 2. the chunk's queries over the cache's first seq_lens[b] + seq tokens
  tk::PrefillParams p{};
  p.q = q; p.k = k_cache; p.v = v_cache; p.out = out; p.out_f32 = out_dtype == TK_F32;
  p.err = dev.err;
  p.B = desc->batch; p.Hq = desc->h_q; p.Hkv = desc->h_kv; p.S = seq; p.R = desc->r;
  p.DV = desc->d_v;
  p.causal = causal != 0;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.num_sms = dev.num_sms;
  p.seq_lens = seq_lens;
  p.page_table = page_table;
  p.k_fmt = key_format(desc->k_dtype);
  p.k_scale = quant ? k_scale : nullptr;
  p.capacity = desc->capacity;
  p.page_size = desc->page_size;
  p.page_shift = a.page_shift;
  p.num_pages = desc->num_pages;
  p.max_pages = desc->max_pages_per_seq;
  p.kv_limit = kv_limit;
  p.kw = quant ? workspace : nullptr;
  p.kw_bytes = quant ? workspace_bytes : 0;
  p.kw_rows = kw_rows;
  e = tk::launch_prefill(p, st, &uns);
  if (uns) return fail(TK_ERR_UNSUPPORTED, "prefill: no kernel for r=%d d_v=%d", desc->r, desc->d_v);
  if (e != cudaSuccess) return cuda_fail(e, "prefill launch");
  return TK_OK;
}

size_t tk_prefill_cached_workspace_size(const tk_cache_desc* desc, int32_t max_seq_len) {
  if (check_desc(desc) != TK_OK || max_seq_len <= 0 || desc->k_dtype == TK_BF16) return 0;
  return tk::prefill_workspace_bytes(desc->batch, desc->h_kv, desc->r, desc->d_v,
                                     key_format(desc->k_dtype), prefill_kw_rows(desc, max_seq_len));
}

size_t tk_decode_workspace_size(const tk_cache_desc* desc, int32_t max_seq_len) {
  if (check_desc(desc) != TK_OK || max_seq_len < 0) return 0;
  DeviceInfo dev;
  if (device_info(&dev) != TK_OK) return 0;
  return tk::plan_decode(desc->batch, desc->h_q, desc->h_kv, desc->r, desc->d_v,
                         key_format(desc->k_dtype), dev.num_sms).bytes;
}

namespace {
tk_status decode_impl(const tk_cache_desc* desc, const void* q, const void* k_cache,
                      const void* v_cache, const float* k_scale, const int32_t* page_table,
                      const int32_t* seq_lens, const void* k_new, const void* v_new,
                      int32_t max_seq_len, void* out, int32_t out_dtype, float scale,
                      void* workspace, size_t workspace_bytes, bool clear_counters,
                      void* stream) {
  const bool fuse = k_new != nullptr || v_new != nullptr;
  tk_status s = check_desc(desc);
  if (s != TK_OK) return s;
  if (max_seq_len < 0) return fail(TK_ERR_INVALID_ARG, "max_seq_len=%d", max_seq_len);
  if (out_dtype != TK_BF16 && out_dtype != TK_F32)
    return fail(TK_ERR_UNSUPPORTED, "out_dtype=%d (supported: TK_BF16, TK_F32)", out_dtype);
  if (!std::isfinite(scale)) return fail(TK_ERR_INVALID_ARG, "scale is not finite");
  if (desc->batch == 0) return TK_OK;
  if ((s = check_cache_ptrs(desc, k_cache, v_cache, k_scale, page_table)) != TK_OK) return s;
  if (!q || !out || !seq_lens) return fail(TK_ERR_INVALID_ARG, "q / out / seq_lens is NULL");
  if (!aligned16(q) || !aligned16(out))
    return fail(TK_ERR_INVALID_ARG, "q / out must be 16-byte aligned");
  if (fuse && (!k_new || !v_new)) return fail(TK_ERR_INVALID_ARG, "k_new / v_new is NULL");
  if (fuse && (!aligned16(k_new) || !aligned16(v_new)))
    return fail(TK_ERR_INVALID_ARG, "k_new / v_new must be 16-byte aligned");
  DeviceInfo dev;
  if ((s = device_info(&dev)) != TK_OK) return s;
  const tk::DecodePlan pl = tk::plan_decode(desc->batch, desc->h_q, desc->h_kv, desc->r, desc->d_v,
                                            key_format(desc->k_dtype), dev.num_sms);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return fail(TK_ERR_WORKSPACE, "workspace is NULL or not 256-byte aligned");
  if (workspace_bytes < pl.bytes)
    return fail(TK_ERR_WORKSPACE, "workspace has %zu bytes, %zu needed", workspace_bytes, pl.bytes);
  unsigned char* ws = static_cast<unsigned char*>(workspace);
  tk::DecodeParams p{};
  p.q = q; p.k = k_cache; p.v = v_cache; p.k_scale = k_scale; p.page_table = page_table;
  p.seq_lens = seq_lens; p.out = out; p.out_f32 = out_dtype == TK_F32;
  p.counters = reinterpret_cast<int32_t*>(ws + pl.off_counters);
  p.part = reinterpret_cast<float*>(ws + pl.off_part);
  p.err = dev.err;
  p.B = desc->batch; p.Hq = desc->h_q; p.Hkv = desc->h_kv; p.R = desc->r; p.DV = desc->d_v;
  p.G = desc->h_q / desc->h_kv;
  p.k_fmt = key_format(desc->k_dtype);
  p.capacity = desc->capacity;
  p.page_size = desc->page_size;
  p.page_shift = desc->page_size ? log2i(desc->page_size) : 0;
  p.num_pages = desc->num_pages; p.max_pages = desc->max_pages_per_seq;
  p.max_seq_len = max_seq_len;
  p.n_cta = pl.n_cta;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.fuse_append = fuse;
  p.k_new = k_new;
  p.v_new = v_new;
  if (clear_counters && tk::decode_max_batch() >= p.B) {
    // every check has passed: zero the arrival counters right before the launch
    const cudaError_t ce = cudaMemsetAsync(p.counters, 0, static_cast<size_t>(p.B) * p.Hkv * sizeof(int32_t),
                                           static_cast<cudaStream_t>(stream));
    if (ce != cudaSuccess) return cuda_fail(ce, "clear arrival counters");
  }
  int uns = 0;
  cudaError_t e = tk::launch_decode(p, static_cast<cudaStream_t>(stream), &uns);
  if (uns) return fail(TK_ERR_UNSUPPORTED, "decode: no kernel for this shape (batch <= %d)",
                       tk::decode_max_batch());
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  return TK_OK;
}
}  // namespace

tk_status tk_attn_decode(const tk_cache_desc* desc, const void* q, const void* k_cache,
                         const void* v_cache, const float* k_scale, const int32_t* page_table,
                         const int32_t* seq_lens, int32_t max_seq_len, void* out,
                         int32_t out_dtype, float scale, void* workspace,
                         size_t workspace_bytes, void* stream) {
  return decode_impl(desc, q, k_cache, v_cache, k_scale, page_table, seq_lens, nullptr, nullptr,
                     max_seq_len, out, out_dtype, scale, workspace, workspace_bytes, false, stream);
}

tk_status tk_attn_decode_append(const tk_cache_desc* desc, const void* q, void* k_cache,
                                void* v_cache, float* k_scale, const int32_t* page_table,
                                const int32_t* seq_lens, const void* k_new, const void* v_new,
                                int32_t max_seq_len, void* out, int32_t out_dtype, float scale,
                                void* workspace, size_t workspace_bytes, void* stream) {
  if (!k_new || !v_new) return fail(TK_ERR_INVALID_ARG, "k_new / v_new is NULL");
  return decode_impl(desc, q, k_cache, v_cache, k_scale, page_table, seq_lens, k_new, v_new,
                     max_seq_len, out, out_dtype, scale, workspace, workspace_bytes, false, stream);
}

}  // extern "C"

namespace tk {
// tk_attn_decode on a caller-supplied scratch whose arrival counters are
// cleared in stream order once every argument check has passed (used by
// tk_attn_decode_noalloc, whose scratch other calls may have left dirty).
tk_status decode_on_scratch(const tk_cache_desc* desc, const void* q, const void* k_cache,
                            const void* v_cache, const float* k_scale, const int32_t* page_table,
                            const int32_t* seq_lens, int32_t max_seq_len, void* out,
                            int32_t out_dtype, float scale, void* scratch, size_t scratch_bytes,
                            void* stream) {
  return decode_impl(desc, q, k_cache, v_cache, k_scale, page_table, seq_lens, nullptr, nullptr,
                     max_seq_len, out, out_dtype, scale, scratch, scratch_bytes, true, stream);
}
}  // namespace tk

extern "C" {

tk_status tk_copy_async(void* dst, const void* src, size_t bytes, void* stream) {
  if (bytes == 0) return TK_OK;
  if (!dst || !src) return fail(TK_ERR_INVALID_ARG, "copy: NULL pointer");
  const cudaError_t e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync");
  return TK_OK;
}

tk_status tk_graph_begin(void* stream) {
  if (!stream) return fail(TK_ERR_INVALID_ARG, "graph capture needs a non-default stream");
  const cudaError_t e = cudaStreamBeginCapture(static_cast<cudaStream_t>(stream),
                                               cudaStreamCaptureModeRelaxed);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamBeginCapture");
  return TK_OK;
}

tk_status tk_graph_end(void* stream, void** graph_out) {
  if (!stream || !graph_out) return fail(TK_ERR_INVALID_ARG, "graph_end: NULL stream or graph_out");
  *graph_out = nullptr;
  cudaGraph_t g = nullptr;
  cudaError_t e = cudaStreamEndCapture(static_cast<cudaStream_t>(stream), &g);
  if (e != cudaSuccess) {
    if (g) cudaGraphDestroy(g);
    return cuda_fail(e, "cudaStreamEndCapture");
  }
  cudaGraphExec_t x = nullptr;
  e = cudaGraphInstantiate(&x, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphInstantiate");
  *graph_out = x;
  return TK_OK;
}

tk_status tk_graph_launch(void* graph, void* stream) {
  if (!graph) return fail(TK_ERR_INVALID_ARG, "graph is NULL");
  const cudaError_t e = cudaGraphLaunch(static_cast<cudaGraphExec_t>(graph), static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphLaunch");
  return TK_OK;
}

tk_status tk_graph_destroy(void* graph) {
  if (!graph) return fail(TK_ERR_INVALID_ARG, "graph is NULL");
  const cudaError_t e = cudaGraphExecDestroy(static_cast<cudaGraphExec_t>(graph));
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphExecDestroy");
  return TK_OK;
}

tk_status tk_check_wait_timeout(int32_t limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 1000000)
    return fail(TK_ERR_INVALID_ARG, "limit_us=%d (1 .. 1000000)", limit_us);
  DeviceInfo dev;
  tk_status s = device_info(&dev);
  if (s != TK_OK) return s;
  const cudaError_t e = tk::launch_wait_timeout(dev.err, static_cast<uint64_t>(limit_us) * 1000u,
                                                static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "wait-timeout check launch");
  return TK_OK;
}

tk_status tk_get_device_error(int32_t* code_out, void* stream) {
  if (!code_out) return fail(TK_ERR_INVALID_ARG, "code_out is NULL");
  DeviceInfo dev;
  tk_status s = device_info(&dev);
  if (s != TK_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int v = 0;
  e = cudaMemcpy(&v, dev.err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "read device error word");
  if (v != 0) {
    const int zero = 0;
    e = cudaMemcpy(dev.err, &zero, sizeof(int), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "clear device error word");
  }
  *code_out = v;
  if (v != 0) return fail(TK_ERR_DEVICE, "device error code %d (%s)", v,
                          v == 1 ? "index out of range" : "wait timed out");
  return TK_OK;
}

const char* tk_status_string(tk_status status) {
  switch (status) {
    case TK_OK: return "TK_OK";
    case TK_ERR_INVALID_ARG: return "TK_ERR_INVALID_ARG";
    case TK_ERR_UNSUPPORTED: return "TK_ERR_UNSUPPORTED";
    case TK_ERR_WORKSPACE: return "TK_ERR_WORKSPACE";
    case TK_ERR_CUDA: return "TK_ERR_CUDA";
    case TK_ERR_DEVICE: return "TK_ERR_DEVICE";
  }
  return "TK_ERR_UNKNOWN";
}

const char* tk_last_error(void) { return t_last_error.c_str(); }

int32_t tk_abi_version(void) { return TK_ABI_VERSION; }

}  // extern "C"
