// quantize.cu — §3.1 quantiser: per-group absmean scale, ternary codes, 2-bit packing,
// zero count per group. One pass over the fp32 latent weights; HBM-bound.
//
// The weight matrix is treated as one flat array: groups (g | k) and code words
// (16 | k) never straddle a row, so group j of row n is flat group n*(k/g)+j and
// the outputs are flat arrays too. One warp owns a unit of 512 consecutive
// weights: four coalesced 16-byte loads per lane, issued before any use. A group
// is reduced with warp shuffles over the g/4 lanes that hold it (g <= 128), or
// over the whole warp and several loads (g = 256, 512). The 32 code words of a
// unit are gathered into lane order and written with one 128-byte store.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace tq {
namespace {

constexpr int kUnit = 512;  // weights per warp per iteration
constexpr int kThreads = 256;

__device__ __forceinline__ uint32_t ternary_code(float w, float s) {
  // Code +-1 iff |fl32(w / s)| > 0.5 (round half to even sends 0.5 to 0 and the
  // clip maps everything beyond 1.5 to +-1). s = 0 gives NaN, hence code 0.
  const float q = __fdiv_rn(w, s);
  return fabsf(q) > 0.5f ? (q < 0.0f ? 3u : 1u) : 0u;
}

template <int G>
__global__ void __launch_bounds__(kThreads) quantize_kernel(const float* __restrict__ w,
                                                            int64_t total,
                                                            uint32_t* __restrict__ codes,
                                                            float* __restrict__ scales,
                                                            int32_t* __restrict__ zeros) {
  static_assert(G == 32 || G == 64 || G == 128 || G == 256 || G == 512, "group size");
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * kThreads) >> 5;
  const int64_t nunits = (total + kUnit - 1) / kUnit;
  constexpr float kInvG = 1.0f / G;  // exact: G is a power of two

  for (int64_t u = warp0; u < nunits; u += nwarps) {
    const int64_t base = u * kUnit;
    float4 v[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t e = base + j * 128 + lane * 4;
      v[j] = e < total ? __ldcs(reinterpret_cast<const float4*>(w + e))
                       : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float part[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      part[j] = (fabsf(v[j].x) + fabsf(v[j].y)) + (fabsf(v[j].z) + fabsf(v[j].w));

    // s = (1/g) * sum |w| for the group holding each chunk of this lane.
    float s[4];
    if constexpr (G <= 128) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float t = part[j];
#pragma unroll
        for (int off = 1; off < G / 4; off <<= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
        s[j] = t * kInvG;
      }
    } else if constexpr (G == 256) {
      float t0 = part[0] + part[1], t1 = part[2] + part[3];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        t0 += __shfl_xor_sync(0xffffffffu, t0, off);
        t1 += __shfl_xor_sync(0xffffffffu, t1, off);
      }
      s[0] = s[1] = t0 * kInvG;
      s[2] = s[3] = t1 * kInvG;
    } else {
      float t = (part[0] + part[1]) + (part[2] + part[3]);
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
      s[0] = s[1] = s[2] = s[3] = t * kInvG;
    }

    // Codes: element i = 4*(lane%4) + e of its 16-code word sits at bit
    // 16*(e&1) + 4*(lane%4) + 2*(e>>1).
    uint32_t word[4];
    int zc[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t c0 = ternary_code(v[j].x, s[j]);
      const uint32_t c1 = ternary_code(v[j].y, s[j]);
      const uint32_t c2 = ternary_code(v[j].z, s[j]);
      const uint32_t c3 = ternary_code(v[j].w, s[j]);
      uint32_t x = (c0 | (c2 << 2) | (c1 << 16) | (c3 << 18)) << (4 * (lane & 3));
      x |= __shfl_xor_sync(0xffffffffu, x, 1);
      x |= __shfl_xor_sync(0xffffffffu, x, 2);
      word[j] = x;
      zc[j] = (c0 == 0) + (c1 == 0) + (c2 == 0) + (c3 == 0);
    }
    // Gather: lane t stores word t of the unit (chunk t/8, lane group t%8).
    uint32_t mine = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t x = __shfl_sync(0xffffffffu, word[j], 4 * (lane & 7));
      if ((lane >> 3) == j) mine = x;
    }
    if (base + lane * 16 < total) codes[(base >> 4) + lane] = mine;

    // Zero counts and scales, one writer per group.
    if constexpr (G <= 128) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        int t = zc[j];
#pragma unroll
        for (int off = 1; off < G / 4; off <<= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
        const int64_t e = base + j * 128 + lane * 4;
        if ((lane & (G / 4 - 1)) == 0 && e < total) {
          scales[e / G] = s[j];
          zeros[e / G] = t;
        }
      }
    } else if constexpr (G == 256) {
      int t0 = zc[0] + zc[1], t1 = zc[2] + zc[3];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        t0 += __shfl_xor_sync(0xffffffffu, t0, off);
        t1 += __shfl_xor_sync(0xffffffffu, t1, off);
      }
      if (lane == 0) {
        scales[base / G] = s[0];
        zeros[base / G] = t0;
        if (base + G < total) {
          scales[base / G + 1] = s[2];
          zeros[base / G + 1] = t1;
        }
      }
    } else {
      int t = (zc[0] + zc[1]) + (zc[2] + zc[3]);
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
      if (lane == 0) {
        scales[base / G] = s[0];
        zeros[base / G] = t;
      }
    }
  }
}

template <int G>
cudaError_t launch(const float* w, int64_t total, uint32_t* codes, float* scales, int32_t* zeros,
                   int num_sms, cudaStream_t stream) {
  const int64_t nunits = (total + kUnit - 1) / kUnit;
  const int64_t warps_per_block = kThreads / 32;
  int64_t blocks = (nunits + warps_per_block - 1) / warps_per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;  // 8 resident blocks per SM
  if (blocks > cap) blocks = cap;
  quantize_kernel<G><<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(w, total, codes,
                                                                           scales, zeros);
  return cudaGetLastError();
}

}  // namespace

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
