// KV-cache append: writes n_new thin-key rows (r wide) and value rows (d_v
// wide) per (sequence, kv head) at logical positions seq_lens[b] + t.
//
// Paper: Section 2.3 (the thin keys k' = x W_K' are what the cache keeps) and
// Section 2.4, Eqs. 8-9 (r + d_v values per token and kv head).  The int8
// variant is the composition with key quantisation of Section 6 (the scheme
// is in kv_row.cuh).
//
// One warp per run of kRows consecutive tokens of one (b, g): every 16-byte
// piece of the run's bf16 rows is loaded before any is stored, so a warp has
// kRows rows in flight (one row per warp leaves the copy far below the HBM
// rate: too few bytes in flight per SM).  Quantised keys take the same
// 16-byte pieces: each lane quantises its 8 elements, and the lanes that hold
// one row (r/8 neighbours) combine their amax by shuffles; the arithmetic per
// element is that of kv_row.cuh's quantiser, so the codes are identical.
#include "common.cuh"
#include "kernels.h"

namespace tk {
namespace {

constexpr int kWarps = 4;
constexpr int kRows = 8;   // tokens per warp

template <int R, int DV, int KF>
__global__ void __launch_bounds__(kWarps * 32) append_kernel(const AppendParams p) {
  const int lane = threadIdx.x & 31;
  const long wg = static_cast<long>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const int n_runs = (p.T + kRows - 1) / kRows;
  const long total = static_cast<long>(p.B) * p.Hkv * n_runs;
  if (wg >= total) return;
  pdl_wait();
  pdl_trigger();
  const int t0 = static_cast<int>(wg % n_runs) * kRows;
  const int g = static_cast<int>((wg / n_runs) % p.Hkv);
  const int b = static_cast<int>(wg / (static_cast<long>(n_runs) * p.Hkv));
  const int pos0 = p.seq_lens[b] + t0;

  // destination row of token t0 + i in the cache / pool, or -1 (past the run's
  // end, or out of range: recorded)
  auto dst_row = [&](int i) -> long long {
    const int pos = pos0 + i;
    if (t0 + i >= p.T) return -1;
    if (p.page_size == 0) {
      if (pos < 0 || pos >= p.capacity) {
        record_error(p.err, TK_DEVERR_INDEX);
        return -1;
      }
      return (static_cast<long long>(b) * p.Hkv + g) * p.capacity + pos;
    }
    const int pidx = pos >> p.page_shift;
    if (pos < 0 || pidx >= p.max_pages) {
      record_error(p.err, TK_DEVERR_INDEX);
      return -1;
    }
    const int page = p.page_table[static_cast<size_t>(b) * p.max_pages + pidx];
    if (page < 0 || page >= p.num_pages) {
      record_error(p.err, TK_DEVERR_INDEX);
      return -1;
    }
    return (static_cast<long long>(page) * p.Hkv + g) * p.page_size + (pos & (p.page_size - 1));
  };
  const size_t src0 = (static_cast<size_t>(b) * p.Hkv + g) * p.T + t0;
  const uint4* vs = static_cast<const uint4*>(p.v_new) + src0 * (2 * DV / 16);
  const uint4* ks = static_cast<const uint4*>(p.k_new) + src0 * (2 * R / 16);
  uint4* vd = static_cast<uint4*>(p.v);
  uint4* kd = static_cast<uint4*>(p.k);
  // values (and bf16 keys): piece c of the run = row c / N, piece c % N of that row
  constexpr int NV = 2 * DV / 16, NK = 2 * R / 16;
  constexpr int PV = (kRows * NV + 31) / 32, PK = (kRows * NK + 31) / 32;
  uint4 vr[PV], kr[PK];
  long long vdst[PV], kdst[PK];
#pragma unroll
  for (int i = 0; i < PV; ++i) {
    const int c = lane + 32 * i;
    vdst[i] = c < kRows * NV ? dst_row(c / NV) : -1;
    if (vdst[i] >= 0) vr[i] = vs[c];
  }
#pragma unroll
  for (int i = 0; i < PK; ++i) {
    const int c = lane + 32 * i;
    kdst[i] = c < kRows * NK ? dst_row(c / NK) : -1;
    if (kdst[i] >= 0) kr[i] = ks[c];
  }
#pragma unroll
  for (int i = 0; i < PV; ++i)
    if (vdst[i] >= 0) vd[vdst[i] * NV + (lane + 32 * i) % NV] = vr[i];
  if constexpr (KF == 0) {
#pragma unroll
    for (int i = 0; i < PK; ++i)
      if (kdst[i] >= 0) kd[kdst[i] * NK + (lane + 32 * i) % NK] = kr[i];
  } else {
    // symmetric per-token quantisation (Section 6): scale = amax / Q (IEEE
    // division), code = clamp(rint(x / scale), -Q, Q), 0 when amax is 0
    constexpr float Q = KF == 1 ? 127.0f : 7.0f;
#pragma unroll
    for (int i = 0; i < PK; ++i) {
      const uint32_t w[4] = {kr[i].x, kr[i].y, kr[i].z, kr[i].w};
      float x[8];
      float amax = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        x[e] = __uint_as_float(e % 2 == 0 ? w[e / 2] << 16 : w[e / 2] & 0xffff0000u);  // bf16 -> f32
        amax = fmaxf(amax, fabsf(x[e]));
      }
      // the NK lanes of one row are neighbours (c = lane + 32 i, NK divides 32)
#pragma unroll
      for (int off = NK / 2; off >= 1; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
      if (kdst[i] < 0) continue;
      const float scale = amax / Q;
      int code[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        float cf = 0.f;
        if (scale != 0.f) cf = fminf(fmaxf(rintf(x[e] / scale), -Q), Q);
        code[e] = static_cast<int>(cf);
      }
      const int piece = (lane + 32 * i) % NK;
      if constexpr (KF == 1) {
        uint2 o;
        o.x = (code[0] & 0xFF) | (code[1] & 0xFF) << 8 | (code[2] & 0xFF) << 16 | (code[3] & 0xFF) << 24;
        o.y = (code[4] & 0xFF) | (code[5] & 0xFF) << 8 | (code[6] & 0xFF) << 16 | (code[7] & 0xFF) << 24;
        *reinterpret_cast<uint2*>(static_cast<int8_t*>(p.k) + kdst[i] * R + piece * 8) = o;
      } else {
        uint32_t o = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) o |= static_cast<uint32_t>(code[e] & 0xF) << (4 * e);
        *reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(p.k) + kdst[i] * (R / 2) + piece * 4) = o;
      }
      if (piece == 0) p.k_scale[kdst[i]] = scale;
    }
  }
}

template <int R, int DV, int KF>
cudaError_t launch_t(const AppendParams& p, cudaStream_t s) {
  const long warps = static_cast<long>(p.B) * p.Hkv * ((p.T + kRows - 1) / kRows);
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
