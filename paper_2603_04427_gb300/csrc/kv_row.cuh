// One warp writes one token's cache row: the r-wide thin key (bf16 copy, or
// int8 codes + fp32 scale) and the d_v-wide value.  Shared by the append
// kernel and the append fused into the decode kernel, so both store the same
// bits.
//
// int8 keys: symmetric absmax per (token, kv head), scale = amax / 127 and
// code = clamp(rint(k / scale), -127, 127), both divisions in IEEE binary32
// (this library is compiled without fast-math); amax 0 stores scale 0 and
// zero codes.  The paper (Section 6) names key quantisation without a
// scheme; this is the library's reading.
#pragma once

#include "common.cuh"

namespace tk {

template <int R, int DV, bool KI8>
__device__ __forceinline__ void write_kv_row(void* k_cache, void* v_cache, float* k_scale,
                                             size_t row, const void* k_src, const void* v_src,
                                             int lane) {
  // values: d_v bf16 = 2 * DV bytes, 16 bytes per lane
  {
    constexpr int NV = 2 * DV / 16;
    const uint4* s = static_cast<const uint4*>(v_src);
    uint4* d = reinterpret_cast<uint4*>(static_cast<unsigned char*>(v_cache) + row * 2 * DV);
    if (lane < NV) d[lane] = s[lane];
  }
  if constexpr (!KI8) {
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
    const float scale = amax / 127.0f;  // IEEE binary32 division
    int8_t* d = static_cast<int8_t*>(k_cache) + row * R;
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      const int c = lane * EPL + e;
      if (c < R) {
        float code = 0.f;
        if (scale != 0.f) code = fminf(fmaxf(rintf(x[e] / scale), -127.f), 127.f);
        d[c] = static_cast<int8_t>(code);
      }
    }
    if (lane == 0) k_scale[row] = scale;
  }
}

}  // namespace tk
