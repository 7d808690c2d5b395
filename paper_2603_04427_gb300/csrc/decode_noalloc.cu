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

#include <mutex>

#include "tk.h"

namespace {

// Scratch for split partials and arrival counters.  Every GPU that loads the
// library holds this array until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[TK_DECODE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
void* g_scratch_ptr[kMaxDevices];
bool g_scratch_ready[kMaxDevices];
std::mutex g_scratch_mu;

// Device address of the scratch array for the current device.  The array's
// name is only a host-side stand-in, so the address is looked up once per
// device, with that device current, and cached.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ready[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = ptr;
    g_scratch_ready[dev] = true;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" tk_status tk_attn_decode_noalloc(const tk_cache_desc* desc, const void* q,
                                            const void* k_cache, const void* v_cache,
                                            const float* k_scale, const int32_t* page_table,
                                            const int32_t* seq_lens, int32_t max_seq_len,
                                            void* out, int32_t out_dtype, float scale,
                                            void* stream) {
  void* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) return TK_ERR_CUDA;
  // 0 means invalid arguments; tk_attn_decode below reports which one.  A need
  // above the scratch size is rejected there as TK_ERR_WORKSPACE ("workspace
  // has N bytes, M needed") before anything is launched.
  const size_t need = tk_decode_workspace_size(desc, max_seq_len);
  if (need != 0 && need <= TK_DECODE_NOALLOC_SCRATCH_BYTES && desc->batch > 0) {
    // The arrival counters (the first batch * h_kv int32 of the scratch) must
    // start at zero.  A completed call leaves them at zero; clearing them in
    // stream order keeps an interrupted earlier call from leaking into this one.
    const size_t counters = static_cast<size_t>(desc->batch) * desc->h_kv * sizeof(int32_t);
    if (cudaMemsetAsync(scratch, 0, counters, static_cast<cudaStream_t>(stream)) != cudaSuccess)
      return TK_ERR_CUDA;
  }
  return tk_attn_decode(desc, q, k_cache, v_cache, k_scale, page_table, seq_lens, max_seq_len,
                        out, out_dtype, scale, scratch, TK_DECODE_NOALLOC_SCRATCH_BYTES, stream);
}
