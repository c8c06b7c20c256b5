// quant_code.cuh — the ternary code word of 16 consecutive weights (§3.1), shared
// by the quantize kernel and the fused AdamW + requantize kernel.
//
// Code decision. The code is +-1 iff fl32(|w| / s) > 0.5 (round half to even sends
// 0.5 to 0; the clip maps everything beyond 1.5 to +-1). The fp32 quotient exceeds
// 0.5 exactly when the real quotient exceeds the midpoint 0.5 + 2^-25 between 0.5
// and its successor, i.e. when |w| > s (1/2 + 2^-25). For a normal s that
// threshold lies strictly between s/2 and the next fp32 value above s/2, so on
// fp32 inputs the test is |w| > s/2 — one comparison reproduces the correctly
// rounded division bit for bit (s/2 is exact for s >= 2^-125). Scales below
// 2^-100 take the division (code_word<true>).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace tq {

// w |= bit when a > h (one compare and one predicated OR).
__device__ __forceinline__ void or_if_gt(uint32_t& w, float a, float h, uint32_t bit) {
  asm("{\n\t.reg .pred p;\n\tsetp.gt.f32 p, %1, %2;\n\t@p or.b32 %0, %0, %3;\n\t}"
      : "+r"(w)
      : "f"(a), "f"(h), "r"(bit));
}

// Code word of 16 consecutive weights; code j at bit p_j = 16*(j&1) + 2*(j>>1),
// high bit the sign, low bit "non-zero".
//   nz:  bit p_j set iff |w_j| > s/2 (fast path) or fl(|w_j| / s) > 0.5.
//   neg: bit p_j + 1 set iff w_j < 0 (sign bit), for every j. The sign bits of
//        weights 2i and 2i+1 (bound for bits 2i+1 and 2i+17) are gathered by one
//        byte permute (bits 15 and 31), one shift and one masked OR.
//   word = nz | (neg & (nz << 1)): the sign only where the code is non-zero.
template <bool kDivide>
__device__ __forceinline__ uint32_t code_word(const float (&x)[16], float s) {
  uint32_t nz = 0, neg = 0;
  if (kDivide) {
#pragma unroll
    for (int j = 0; j < 16; ++j)
      or_if_gt(nz, fabsf(__fdiv_rn(x[j], s)), 0.5f, 1u << (16 * (j & 1) + 2 * (j >> 1)));
  } else {
    const float h = 0.5f * s;
#pragma unroll
    for (int j = 0; j < 16; ++j) or_if_gt(nz, fabsf(x[j]), h, 1u << (16 * (j & 1) + 2 * (j >> 1)));
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t hi = __byte_perm(__float_as_uint(x[2 * i]), __float_as_uint(x[2 * i + 1]), 0x7632);
    neg |= (hi >> (14 - 2 * i)) & ((1u << (2 * i + 1)) | (1u << (2 * i + 17)));
  }
  return nz | (neg & (nz << 1));
}

// Code word against a caller-given scale of either sign (the learnable-scale
// variant): c = round(clip(w / s)). For s < 0 the fp32 quotient of the negated
// operands is the same number, so the word is that of -w against -s; scales below
// 2^-100 (zero, denormal) or NaN-free tiny values take the division. Every lane in
// `live` must call it.
__device__ __forceinline__ uint32_t code_word_any(const float (&x)[16], float s, unsigned live) {
  const bool flip = s < 0.f;
  const float t = flip ? -s : s;
  float y[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) y[j] = flip ? -x[j] : x[j];
  const bool tiny = t < 0x1p-100f;
  return __any_sync(live, tiny) ? (tiny ? code_word<true>(y, t) : code_word<false>(y, t))
                                : code_word<false>(y, t);
}

}  // namespace tq
