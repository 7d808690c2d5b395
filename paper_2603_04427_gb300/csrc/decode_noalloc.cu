// Decode entry point for callers that cannot allocate device memory.
//
// tk_attn_decode needs a caller-provided workspace for the per-split partial
// results and the per-(sequence, kv head) arrival counters.  Some callers have
// no way to obtain one: an inference runtime whose device memory is fully
// pre-reserved by its own pool and that forbids cudaMalloc on the decode path
// (it synchronises the device and can fail under fragmentation), plugin hosts
// that hand a plugin only its inputs and outputs, and real-time loops that must
// not touch the allocator between steps.  tk_attn_decode_noalloc serves them
// from a fixed scratch array that lives in this library's device image.
//
// The paper has no counterpart to this entry point; it is an interface
// convenience around the same decode kernel.
#include <cuda_runtime.h>

#include "tk.h"

namespace tk {
tk_status decode_on_scratch(const tk_cache_desc* desc, const void* q, const void* k_cache,
                            const void* v_cache, const float* k_scale, const int32_t* page_table,
                            const int32_t* seq_lens, int32_t max_seq_len, void* out,
                            int32_t out_dtype, float scale, void* scratch, size_t scratch_bytes,
                            void* stream);
}  // namespace tk

namespace {

// Scratch for split partials and arrival counters.  Every GPU that loads the
// library holds this array until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[TK_DECODE_NOALLOC_SCRATCH_BYTES];

}  // namespace

extern "C" tk_status tk_attn_decode_noalloc(const tk_cache_desc* desc, const void* q,
                                            const void* k_cache, const void* v_cache,
                                            const float* k_scale, const int32_t* page_table,
                                            const int32_t* seq_lens, int32_t max_seq_len,
                                            void* out, int32_t out_dtype, float scale,
                                            void* stream) {
  // The array's name is only a host-side stand-in: its device address is
  // looked up with the calling thread's current device, on every call
  // (cudaGetSymbolAddress allocates nothing), so that an address from before
  // a cudaDeviceReset is never reused.
  void* scratch = nullptr;
  if (cudaGetSymbolAddress(&scratch, g_noalloc_scratch) != cudaSuccess) return TK_ERR_CUDA;
  // tk_attn_decode's checks run first; a shape whose workspace need exceeds
  // the array is rejected as TK_ERR_WORKSPACE ("workspace has N bytes, M
  // needed") and a rejected call writes nothing.  Only a call that passed
  // every check clears the arrival counters (the first batch * h_kv int32 of
  // the scratch) in stream order, right before its launch.
  return tk::decode_on_scratch(desc, q, k_cache, v_cache, k_scale, page_table, seq_lens,
                               max_seq_len, out, out_dtype, scale, scratch,
                               TK_DECODE_NOALLOC_SCRATCH_BYTES, stream);
}
