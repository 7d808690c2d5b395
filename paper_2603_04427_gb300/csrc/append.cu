// KV-cache append: writes n_new thin-key rows (r wide) and value rows (d_v
// wide) per (sequence, kv head) at logical positions seq_lens[b] + t.
//
// Paper: Section 2.3 (the thin keys k' = x W_K' are what the cache keeps) and
// Section 2.4, Eqs. 8-9 (r + d_v values per token and kv head).  The int8
// variant is the composition with key quantisation of Section 6 (the scheme
// is in kv_row.cuh).
//
// One warp per (b, g, t): 16-byte vector loads and stores for bf16 rows; for
// int8 keys a warp max-reduction gives amax.
#include "common.cuh"
#include "kernels.h"
#include "kv_row.cuh"

namespace tk {
namespace {

constexpr int kWarps = 4;

template <int R, int DV, int KF>
__global__ void __launch_bounds__(kWarps * 32) append_kernel(const AppendParams p) {
  const int lane = threadIdx.x & 31;
  const long wg = static_cast<long>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const long total = static_cast<long>(p.B) * p.Hkv * p.T;
  if (wg >= total) return;
  pdl_wait();
  pdl_trigger();
  const int t = static_cast<int>(wg % p.T);
  const int g = static_cast<int>((wg / p.T) % p.Hkv);
  const int b = static_cast<int>(wg / (static_cast<long>(p.T) * p.Hkv));
  const int pos = p.seq_lens[b] + t;

  size_t row;  // destination row in the cache / pool
  if (p.page_size == 0) {
    if (pos < 0 || pos >= p.capacity) {
      if (lane == 0) record_error(p.err, TK_DEVERR_INDEX);
      return;
    }
    row = (static_cast<size_t>(b) * p.Hkv + g) * p.capacity + pos;
  } else {
    const int pidx = pos >> p.page_shift;
    if (pos < 0 || pidx >= p.max_pages) {
      if (lane == 0) record_error(p.err, TK_DEVERR_INDEX);
      return;
    }
    const int page = p.page_table[static_cast<size_t>(b) * p.max_pages + pidx];
    if (page < 0 || page >= p.num_pages) {
      if (lane == 0) record_error(p.err, TK_DEVERR_INDEX);
      return;
    }
    row = (static_cast<size_t>(page) * p.Hkv + g) * p.page_size + (pos & (p.page_size - 1));
  }
  const size_t src = (static_cast<size_t>(b) * p.Hkv + g) * p.T + t;
  write_kv_row<R, DV, KF>(p.k, p.v, p.k_scale, row,
                           static_cast<const unsigned char*>(p.k_new) + src * 2 * R,
                           static_cast<const unsigned char*>(p.v_new) + src * 2 * DV, lane);
}

template <int R, int DV, int KF>
cudaError_t launch_t(const AppendParams& p, cudaStream_t s) {
  const long warps = static_cast<long>(p.B) * p.Hkv * p.T;
  const long blocks = (warps + kWarps - 1) / kWarps;
  if (blocks > 0x7fffffffL) return cudaErrorInvalidConfiguration;
  return launch_pdl(append_kernel<R, DV, KF>, dim3(static_cast<unsigned>(blocks)),
                    dim3(kWarps * 32), 0, s, p);
}

template <int R, int KF>
cudaError_t by_dv(const AppendParams& p, cudaStream_t s, int* uns) {
  switch (p.DV) {
    case 64: return launch_t<R, 64, KF>(p, s);
    case 128: return launch_t<R, 128, KF>(p, s);
  }
  *uns = 1;
  return cudaSuccess;
}

template <int KF>
cudaError_t by_r(const AppendParams& p, cudaStream_t s, int* uns) {
  switch (p.R) {
    case 16:
      if constexpr (KF != 2) return by_dv<16, KF>(p, s, uns);
      break;  // int4 keys need r >= 32
    case 32: return by_dv<32, KF>(p, s, uns);
    case 64: return by_dv<64, KF>(p, s, uns);
    case 128: return by_dv<128, KF>(p, s, uns);
  }
  *uns = 1;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_append(const AppendParams& p, cudaStream_t stream, int* unsupported) {
  *unsupported = 0;
  if (p.T == 0 || p.B == 0) return cudaSuccess;
  switch (p.k_fmt) {
    case 0: return by_r<0>(p, stream, unsupported);
    case 1: return by_r<1>(p, stream, unsupported);
    case 2: return by_r<2>(p, stream, unsupported);
  }
  *unsupported = 1;
  return cudaSuccess;
}

}  // namespace tk
