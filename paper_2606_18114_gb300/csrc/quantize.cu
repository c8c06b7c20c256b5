// quantize.cu — §3.1 quantiser: per-group absmean scale, ternary codes, 2-bit packing,
// zero count per group. One pass over the fp32 latent weights; HBM-bound.
//
// The weight matrix is treated as one flat array: groups (g | k) and code words
// (16 | k) never straddle a row, so group j of row n is flat group n*(k/g)+j and
// the outputs are flat arrays too. Each lane owns 16 consecutive weights — one
// code word — read as four 16-byte loads; a warp covers 512 weights per unit and
// keeps two units of loads in flight. A group spans g/16 consecutive lanes and is
// reduced with log2(g/16) xor-shuffles; the zero count of a word is
// 16 - popc(word & 0x5555...) because every non-zero code has its low bit set.
//
// Code decision. The code is +-1 iff fl32(|w| / s) > 0.5 (round half to even sends
// 0.5 to 0; the clip maps everything beyond 1.5 to +-1). The fp32 quotient exceeds
// 0.5 exactly when the real quotient exceeds the midpoint 0.5 + 2^-25 between 0.5
// and its successor, i.e. when |w| - s/2 > s * 2^-25. For s >= 2^-100 both s/2
// and s * 2^-25 are exact, and |w| - s/2 is exact whenever s/4 <= |w| <= s
// (Sterbenz); outside that band its rounded value still has the right side of
// the threshold. So one fused multiply-add and one compare reproduce the
// correctly rounded division bit for bit. Smaller scales take the division.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace tq {
namespace {

constexpr int kUnit = 512;    // weights per warp per unit
constexpr int kUnroll = 2;    // units per warp iteration (loads in flight)
constexpr int kThreads = 256;

__device__ __forceinline__ uint32_t code_bits(float w, float s, float t, bool tiny_s) {
  const bool nz = tiny_s ? fabsf(__fdiv_rn(w, s)) > 0.5f : __fmaf_rn(-0.5f, s, fabsf(w)) > t;
  const uint32_t neg = __float_as_uint(w) >> 31;
  return nz ? (1u | (neg << 1)) : 0u;
}

template <int G>
__global__ void __launch_bounds__(kThreads) quantize_kernel(const float* __restrict__ w,
                                                            int64_t total,
                                                            uint32_t* __restrict__ codes,
                                                            float* __restrict__ scales,
                                                            int32_t* __restrict__ zeros) {
  static_assert(G == 32 || G == 64 || G == 128 || G == 256 || G == 512, "group size");
  constexpr int kLanesPerGroup = G / 16;
  constexpr float kInvG = 1.0f / G;  // exact: G is a power of two
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int64_t nunits = (total + kUnit - 1) / kUnit;

  for (int64_t u0 = warp0 * kUnroll; u0 < nunits; u0 += nwarps * kUnroll) {
    float4 v[kUnroll][4];
#pragma unroll
    for (int r = 0; r < kUnroll; ++r) {
      const int64_t e = (u0 + r) * kUnit + lane * 16;
      const bool in = e < total;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        v[r][j] = in ? __ldg(reinterpret_cast<const float4*>(w + e) + j)
                     : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int r = 0; r < kUnroll; ++r) {
      const int64_t e = (u0 + r) * kUnit + lane * 16;
      float sum = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        sum += (fabsf(v[r][j].x) + fabsf(v[r][j].y)) + (fabsf(v[r][j].z) + fabsf(v[r][j].w));
#pragma unroll
      for (int off = 1; off < kLanesPerGroup; off <<= 1)
        sum += __shfl_xor_sync(0xffffffffu, sum, off);
      const float s = sum * kInvG;            // s = (1/g) * sum |w|
      const float t = s * 0x1p-25f;           // half an ulp of 0.5, in units of s
      const bool tiny = s < 0x1p-100f;
      const float x[16] = {v[r][0].x, v[r][0].y, v[r][0].z, v[r][0].w,
                           v[r][1].x, v[r][1].y, v[r][1].z, v[r][1].w,
                           v[r][2].x, v[r][2].y, v[r][2].z, v[r][2].w,
                           v[r][3].x, v[r][3].y, v[r][3].z, v[r][3].w};
      uint32_t word = 0;
#pragma unroll
      for (int i = 0; i < 16; ++i)  // code i at bit 16*(i&1) + 2*(i>>1)
        word |= code_bits(x[i], s, t, tiny) << (16 * (i & 1) + 2 * (i >> 1));
      int zc = 16 - __popc(word & 0x55555555u);
#pragma unroll
      for (int off = 1; off < kLanesPerGroup; off <<= 1) zc += __shfl_xor_sync(0xffffffffu, zc, off);
      if (e < total) {
        codes[e >> 4] = word;
        if ((lane & (kLanesPerGroup - 1)) == 0) {
          scales[e / G] = s;
          zeros[e / G] = zc;
        }
      }
    }
  }
}

template <int G>
cudaError_t launch(const float* w, int64_t total, uint32_t* codes, float* scales, int32_t* zeros,
                   int num_sms, cudaStream_t stream) {
  const int64_t nunits = (total + kUnit - 1) / kUnit;
  const int64_t warps_needed = (nunits + kUnroll - 1) / kUnroll;
  const int64_t warps_per_block = kThreads / 32;
  int64_t blocks = (warps_needed + warps_per_block - 1) / warps_per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;  // 8 resident blocks per SM
  if (blocks > cap) blocks = cap;
  quantize_kernel<G><<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(w, total, codes,
                                                                           scales, zeros);
  return cudaGetLastError();
}

// codes [n][k/16] -> codes_t [k][ldt]: a 128 x 128 (n x k) tile per block. The tile's
// 128 rows x 8 code words are read with one 32-byte sector per row, and each
// output row k receives 8 consecutive words (one sector) of the transposed tile.
__device__ __forceinline__ int code_pos(int i) { return 16 * (i & 1) + 2 * (i >> 1); }

__global__ void __launch_bounds__(256) transpose_codes_kernel(const uint32_t* __restrict__ codes,
                                                              int64_t n, int64_t k,
                                                              uint32_t* __restrict__ codes_t,
                                                              int64_t ldt) {
  __shared__ uint32_t tile[128][9];
  const int64_t n0 = static_cast<int64_t>(blockIdx.y) * 128;
  const int64_t k0 = static_cast<int64_t>(blockIdx.x) * 128;
  const int64_t words = k >> 4;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = threadIdx.x + 256 * i;
    const int r = idx >> 3, c = idx & 7;
    const int64_t row = n0 + r, col = (k0 >> 4) + c;
    tile[r][c] = (row < n && col < words) ? codes[row * words + col] : 0u;
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = threadIdx.x + 256 * i;
    const int kk = idx >> 3, ww = idx & 7;
    const int64_t kg = k0 + kk, wg = (n0 >> 4) + ww;
    if (kg >= k || wg >= ldt) continue;
    const int c = kk >> 4, sh = code_pos(kk & 15);
    uint32_t out = 0;
#pragma unroll
    for (int j = 0; j < 16; ++j) out |= ((tile[16 * ww + j][c] >> sh) & 3u) << code_pos(j);
    codes_t[kg * ldt + wg] = out;
  }
}

}  // namespace

cudaError_t launch_transpose_codes(const uint32_t* codes, int64_t n, int64_t k, uint32_t* codes_t,
                                   cudaStream_t stream) {
  const int64_t ldt = 4 * ((n + 63) / 64);
  dim3 grid(static_cast<unsigned>((k + 127) / 128), static_cast<unsigned>((n + 127) / 128));
  transpose_codes_kernel<<<grid, 256, 0, stream>>>(codes, n, k, codes_t, ldt);
  return cudaGetLastError();
}

cudaError_t launch_quantize(const float* w, int64_t n, int64_t k, int g, uint32_t* codes,
                            float* scales, int32_t* zeros, int num_sms, cudaStream_t stream) {
  const int64_t total = n * k;
  switch (g) {
    case 32: return launch<32>(w, total, codes, scales, zeros, num_sms, stream);
    case 64: return launch<64>(w, total, codes, scales, zeros, num_sms, stream);
    case 128: return launch<128>(w, total, codes, scales, zeros, num_sms, stream);
    case 256: return launch<256>(w, total, codes, scales, zeros, num_sms, stream);
    case 512: return launch<512>(w, total, codes, scales, zeros, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace tq
