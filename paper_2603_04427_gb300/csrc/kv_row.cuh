// One warp writes one token's cache row: the r-wide thin key (bf16 copy, or
// int8 / int4 codes + fp32 scale) and the d_v-wide value.  Shared by the
// append kernel and the append fused into the decode kernel, so both store
// the same bits.
//
// Quantised keys: symmetric absmax per (token, kv head), scale = amax / Q and
// code = clamp(rint(k / scale), -Q, Q) with Q = 127 (int8) or 7 (int4), both
// divisions in IEEE binary32 (this library is compiled without fast-math);
// amax 0 stores scale 0 and zero codes.  int4 codes are stored two per byte,
// element 2j in bits 0-3 and 2j+1 in bits 4-7 (4-bit two's complement).  The
// paper (Section 6) names key quantisation and its 4-bit composition without
// a scheme; this is the library's reading.
#pragma once

#include "common.cuh"

namespace tk {

// The value row: d_v bf16 = 2 * DV bytes, 16 bytes per lane.
template <int DV>
__device__ __forceinline__ void write_v_row(void* v_cache, size_t row, const void* v_src, int lane) {
  constexpr int NV = 2 * DV / 16;
  const uint4* s = static_cast<const uint4*>(v_src);
  uint4* d = reinterpret_cast<uint4*>(static_cast<unsigned char*>(v_cache) + row * 2 * DV);
  if (lane < NV) d[lane] = s[lane];
}

// The key row.  KF: key format, 0 bf16, 1 int8, 2 int4 (R >= 32).
template <int R, int KF>
__device__ __forceinline__ void write_k_row(void* k_cache, float* k_scale, size_t row,
                                            const void* k_src, int lane) {
  if constexpr (KF == 0) {
    constexpr int NK = 2 * R / 16;
    const uint4* s = static_cast<const uint4*>(k_src);
    uint4* d = reinterpret_cast<uint4*>(static_cast<unsigned char*>(k_cache) + row * 2 * R);
    if (lane < NK) d[lane] = s[lane];
  } else {
    // each lane holds EPL = ceil(R / 32) consecutive key elements
    constexpr int EPL = R >= 32 ? R / 32 : 1;
    const __nv_bfloat16* s = static_cast<const __nv_bfloat16*>(k_src);
    float x[EPL];
    float amax = 0.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      const int c = lane * EPL + e;
      x[e] = c < R ? __bfloat162float(s[c]) : 0.f;
      amax = fmaxf(amax, fabsf(x[e]));
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
    constexpr float Q = KF == 1 ? 127.0f : 7.0f;
    const float scale = amax / Q;  // IEEE binary32 division
    int code[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      float cf = 0.f;
      if (scale != 0.f) cf = fminf(fmaxf(rintf(x[e] / scale), -Q), Q);
      code[e] = static_cast<int>(cf);
    }
    if constexpr (KF == 1) {
      int8_t* d = static_cast<int8_t*>(k_cache) + row * R;
#pragma unroll
      for (int e = 0; e < EPL; ++e) {
        const int c = lane * EPL + e;
        if (c < R) d[c] = static_cast<int8_t>(code[e]);
      }
    } else {
      static_assert(R >= 32, "int4 keys need r >= 32");
      uint8_t* d = static_cast<uint8_t*>(k_cache) + row * (R / 2);
      if constexpr (EPL == 1) {
        // element `lane`; the even lane packs itself with its odd neighbour
        const int hi = __shfl_down_sync(0xffffffffu, code[0], 1);
        if ((lane & 1) == 0) d[lane / 2] = static_cast<uint8_t>((code[0] & 0xF) | ((hi & 0xF) << 4));
      } else {
#pragma unroll
        for (int e = 0; e < EPL; e += 2)
          d[(lane * EPL + e) / 2] = static_cast<uint8_t>((code[e] & 0xF) | ((code[e + 1] & 0xF) << 4));
      }
    }
    if (lane == 0) k_scale[row] = scale;
  }
}

// The whole cache row of one token: value, then key.
template <int R, int DV, int KF>
__device__ __forceinline__ void write_kv_row(void* k_cache, void* v_cache, float* k_scale,
                                             size_t row, const void* k_src, const void* v_src,
                                             int lane) {
  write_v_row<DV>(v_cache, row, v_src, lane);
  write_k_row<R, KF>(k_cache, k_scale, row, k_src, lane);
}

}  // namespace tk
