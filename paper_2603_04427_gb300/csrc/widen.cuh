// Exact widening of quantised key codes to bf16 pairs, shared by the decode
// and chunked-prefill kernels.  Integer-to-float conversion instructions run
// on the same unit as ex2 (the softmax's exponentials); these use integer
// byte moves and one fp32 or bf16 subtraction instead.
#pragma once

#include "common.cuh"

namespace tk {

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
// Four int8 (one 32-bit word) to two bf16 pairs, exactly: each byte (biased by
// 128) becomes the low mantissa byte of 2^23, and 2^23 + 128 is subtracted.
__device__ __forceinline__ void i8x4_to_bf16(uint32_t w, uint32_t& lo, uint32_t& hi) {
  const uint32_t x = w ^ 0x80808080u;
  uint32_t f0, f1, f2, f3;
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7540;" : "=r"(f0) : "r"(x));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7541;" : "=r"(f1) : "r"(x));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7542;" : "=r"(f2) : "r"(x));
  asm("prmt.b32 %0, %1, 0x4B000000, 0x7543;" : "=r"(f3) : "r"(x));
  const float bias = 8388736.0f;  // 2^23 + 128
  lo = pack_bf16(__uint_as_float(f0) - bias, __uint_as_float(f1) - bias);
  hi = pack_bf16(__uint_as_float(f2) - bias, __uint_as_float(f3) - bias);
}
// Eight int4 codes (one 32-bit word, code i in bits 4i..4i+3, 4-bit two's
// complement) to four bf16 pairs (codes 0,1), (2,3), (4,5), (6,7), exactly:
// flipping each code's sign bit gives c + 8 in [0, 15], which becomes the low
// mantissa bits of bf16 128 (128 + c + 8), and 136 is subtracted.
__device__ __forceinline__ uint32_t bf16x2_minus136(uint32_t x) {
  uint32_t d;
  asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(x), "r"(0x43084308u));
  return d;
}
__device__ __forceinline__ void i4x8_to_bf16(uint32_t w, uint32_t& p01, uint32_t& p23,
                                             uint32_t& p45, uint32_t& p67) {
  const uint32_t x = w ^ 0x88888888u;
  const uint32_t k = 0x43004300u;  // bf16 128.0 in both halves
  p01 = bf16x2_minus136(k | (x & 0xFu) | ((x << 12) & 0xF0000u));
  p23 = bf16x2_minus136(k | ((x >> 8) & 0xFu) | ((x << 4) & 0xF0000u));
  p45 = bf16x2_minus136(k | ((x >> 16) & 0xFu) | ((x >> 4) & 0xF0000u));
  p67 = bf16x2_minus136(k | ((x >> 24) & 0xFu) | ((x >> 12) & 0xF0000u));
}

}  // namespace tk
