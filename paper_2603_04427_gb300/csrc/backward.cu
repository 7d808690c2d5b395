// Backward pass of thin-key attention (the training path): dQ and dK are r
// wide, dV is d_v wide.
//
// Paper: Section 2.1, Eqs. 1-4 (the forward being differentiated); training
// with thin keys is Sections 3.2-3.3.  Per head, with s = scale q k^T (masked),
// p = softmax(s), out = p v and dL/d(out) = dO:
//     dV = p^T dO,   dP = dO v^T,   dS = p * (dP - D),  D_i = sum_c dO_ic out_ic,
//     dQ = scale dS k,   dK = scale dS^T q
// (D_i equals rowsum(dP * p) for the exact forward output).
//
// Two kernels: bwd_prep below (-D = -rowsum(dO * out) and -lse log2(e) per
// query row, rows padded to a multiple of 128, and dQ set to zero), then the
// tensor-memory gradient kernel of backward_tc.cu.
#include <cuda_bf16.h>

#include "common.cuh"
#include "kernels.h"

namespace tk {
namespace {

// ---------------------------------------------------------------- preprocessing
// DV / 8 threads per padded statistics row (b, h, i < S_pad), 16 bytes of out
// and of d_out each: for i < S, nd = -sum_c dO * out (fp32), nl2 = -lse *
// log2(e) and the row of dQ zeroed; for S <= i < S_pad, nd = 0 and nl2 = -inf
// (such rows get softmax weight 0).
constexpr int kPrepThreads = 256;
template <int R, int DV>
__global__ void __launch_bounds__(kPrepThreads) bwd_prep(const BackwardParams p) {
  constexpr int TPR = DV / 8;                       // threads per row
  constexpr int RPB = kPrepThreads / TPR;           // rows per block
  static_assert(32 % TPR == 0, "a row's threads sit in one warp");
  const int sub = threadIdx.x % TPR;
  const long long row = static_cast<long long>(blockIdx.x) * RPB + threadIdx.x / TPR;
  const long long rows = static_cast<long long>(p.B) * p.Hq * p.S_pad;
  // no lane leaves before the shuffle below: a warp holds several rows
  const bool in_grid = row < rows;
  const long long bh = in_grid ? row / p.S_pad : 0;
  const int i = in_grid ? static_cast<int>(row - bh * p.S_pad) : 0;
  const bool real = in_grid && i < p.S;
  const long long x = bh * p.S + i;   // row of the [B][Hq][S] tensors
  float acc = 0.f;
  if (real) {
    const uint4 o = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.out) + x * DV)[sub];
    const uint4 d = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.d_out) + x * DV)[sub];
    const uint32_t ow[4] = {o.x, o.y, o.z, o.w}, dw[4] = {d.x, d.y, d.z, d.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) acc += bf16lo(ow[e]) * bf16lo(dw[e]) + bf16hi(ow[e]) * bf16hi(dw[e]);
  }
#pragma unroll
  for (int off = TPR / 2; off >= 1; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (!in_grid) return;
  if (sub == 0) {
    p.nd[row] = real ? -acc : 0.f;
    p.nl2[row] = real ? -p.lse[x] * 1.4426950408889634f : -INFINITY;
  }
  if (!real) return;
  float4* dq = reinterpret_cast<float4*>(p.dq + x * R);
#pragma unroll
  for (int c = sub; c < R / 4; c += TPR) dq[c] = make_float4(0.f, 0.f, 0.f, 0.f);
}

template <int R, int DV>
cudaError_t launch_t(const BackwardParams& p, cudaStream_t s, int* uns) {
  const long long rows = static_cast<long long>(p.B) * p.Hq * p.S_pad;
  constexpr int rpb = kPrepThreads / (DV / 8);
  const long long pblocks = (rows + rpb - 1) / rpb;
  if (pblocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  bwd_prep<R, DV><<<static_cast<unsigned>(pblocks), kPrepThreads, 0, s>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_backward_tc(p, s, uns);
}

template <int R>
cudaError_t by_dv(const BackwardParams& p, cudaStream_t s, int* uns) {
  switch (p.DV) {
    case 64: return launch_t<R, 64>(p, s, uns);
    case 128: return launch_t<R, 128>(p, s, uns);
  }
  *uns = 1;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_backward(const BackwardParams& p, cudaStream_t stream, int* unsupported) {
  *unsupported = 0;
  switch (p.R) {
    case 16: return by_dv<16>(p, stream, unsupported);
    case 32: return by_dv<32>(p, stream, unsupported);
    case 64: return by_dv<64>(p, stream, unsupported);
    case 128: return by_dv<128>(p, stream, unsupported);
  }
  *unsupported = 1;
  return cudaSuccess;
}

}  // namespace tk
