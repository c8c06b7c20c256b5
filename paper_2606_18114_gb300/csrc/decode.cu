// decode.cu — W1.58A16 forward for few tokens (m <= 16): an HBM-streaming kernel
// over the packed codes of one or many matrices in one launch (§8: at small batch
// the layer is bound by weight traffic; 2-bit codes + fp32 group scales are 0.28
// bytes per weight at g = 128).
//
// Work unit = 16 consecutive weight rows of one matrix over its whole K; each warp
// walks units u = global_warp, global_warp + warps, ... across all matrices.
// Per 64-wide chunk of K a warp runs four mma.sync.m16n8k16 (bf16 in, fp32
// accumulate) with the expanded weights as the 16 x 16 A operand and up to 8
// tokens as the n8 B operand (two B tiles for 9..16 tokens).
//
// The reduction index of the MMA is permuted identically on both operands so that
// lane (g, t) (g = lane / 4, t = lane % 4) consumes exactly code word t of the
// chunk for rows g and g + 8 — reduction offsets 16t .. 16t + 15 — and the
// contiguous 32 bytes x[token g][16t .. 16t + 15]: MMA number kb of the chunk
// uses offsets 16t + 4kb + {0,1} for fragment slots (2t, 2t+1) and 16t + 4kb +
// {2,3} for slots (2t+8, 2t+9). Code words and x are then read with coalesced
// loads and no lane reads what another lane reads.
//
// Expansion: pair j of a code word -> bf16x2 (2c, 2c) by ((w << (14 - 2j)) &
// 0xC000C000) (layout of include/tq.h). For g >= 64 every chunk lies in one group,
// so partial sums of a group are scaled by s/2 in fp32 (exact scale); for g = 32 the
// two groups of a chunk meet inside one MMA, so the expansion multiplies by
// bf16(s)/2 as the prefill kernels do.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace tq {
namespace {

constexpr int kThreads = 256;
constexpr int kPrefetch = 6;   // chunks of code words in flight per warp

__device__ __forceinline__ uint32_t bmul2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

__device__ __forceinline__ uint32_t pair_bits(uint32_t w, int j) {
  return (w << (14 - 2 * j)) & 0xC000C000u;
}

__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t ldg_nc(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

__device__ __forceinline__ uint32_t half_scale_bf16x2(float s) {
  const __nv_bfloat16 h = __float2bfloat16_rn(0.5f * s);
  const uint32_t u = __bfloat16_as_ushort(h);
  return u | (u << 16);
}

// Binary search: matrix d with unit0[d] <= u < unit0[d + 1].
__device__ __forceinline__ int find_mat(const DecodeBatch& b, int u) {
  int lo = 0, hi = b.count - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (b.mats[mid].unit0 <= u) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <bool kTwoTiles>
__global__ void __launch_bounds__(kThreads, 3) decode_kernel(const __grid_constant__ DecodeBatch b) {
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int gwarp = static_cast<int>((blockIdx.x * kThreads + threadIdx.x) >> 5);
  const int nwarps = static_cast<int>((gridDim.x * kThreads) >> 5);
  const int m = b.m;

  for (int u = gwarp; u < b.total_units; u += nwarps) {
    const int d = find_mat(b, u);
    const DecodeMat& mat = b.mats[d];
    const int64_t n = mat.n, k = mat.k;
    const int64_t r0 = static_cast<int64_t>(u - mat.unit0) * 16;
    const int64_t words = k >> 4;                  // code words per row
    const int nchunk = static_cast<int>(k >> 6);   // 64-wide chunks
    const int64_t ra = r0 + g, rb = r0 + g + 8;    // this lane's two rows
    const bool va = ra < n, vb = rb < n;
    const uint32_t* ca = mat.codes + ra * words + t;
    const uint32_t* cb = mat.codes + rb * words + t;
    const int log2g = mat.log2g;
    const int64_t gpr = k >> log2g;
    const float* sa = mat.scales + ra * gpr;
    const float* sb = mat.scales + rb * gpr;
    // x rows of this lane's tokens (g and g + 8); tokens >= m read as zeros
    const __nv_bfloat16* xa = static_cast<const __nv_bfloat16*>(mat.x) + static_cast<int64_t>(g) * k + 16 * t;
    const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(mat.x) + static_cast<int64_t>(g + 8) * k + 16 * t;
    const bool ta = g < m, tb = kTwoTiles && (g + 8 < m);

    // code words of the first chunks
    uint32_t qa[kPrefetch], qb[kPrefetch];
#pragma unroll
    for (int p = 0; p < kPrefetch; ++p) {
      qa[p] = (va && p < nchunk) ? ldg_nc(ca + 4 * p) : 0u;
      qb[p] = (vb && p < nchunk) ? ldg_nc(cb + 4 * p) : 0u;
    }

    float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
    float part0[4] = {0.f, 0.f, 0.f, 0.f}, part1[4] = {0.f, 0.f, 0.f, 0.f};
    const int chunks_per_group = log2g >= 6 ? (1 << (log2g - 6)) : 1;

    for (int c0 = 0; c0 < nchunk; c0 += kPrefetch) {
#pragma unroll
      for (int p = 0; p < kPrefetch; ++p) {
        const int c = c0 + p;
        if (c >= nchunk) break;
        const uint32_t wa = qa[p], wb = qb[p];
        const int cn = c + kPrefetch;  // refill this slot
        qa[p] = (va && cn < nchunk) ? ldg_nc(ca + 4 * cn) : 0u;
        qb[p] = (vb && cn < nchunk) ? ldg_nc(cb + 4 * cn) : 0u;
        // x fragments: 32 contiguous bytes per token row
        uint4 x0 = make_uint4(0, 0, 0, 0), x1 = make_uint4(0, 0, 0, 0);
        uint4 y0 = make_uint4(0, 0, 0, 0), y1 = make_uint4(0, 0, 0, 0);
        if (ta) {
          x0 = __ldg(reinterpret_cast<const uint4*>(xa + 64 * c));
          x1 = __ldg(reinterpret_cast<const uint4*>(xa + 64 * c + 8));
        }
        if (tb) {
          y0 = __ldg(reinterpret_cast<const uint4*>(xb + 64 * c));
          y1 = __ldg(reinterpret_cast<const uint4*>(xb + 64 * c + 8));
        }
        const uint32_t xr[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
        const uint32_t yr[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
        if (log2g == 5) {
          // g = 32: lane t's offsets 16t..16t+15 lie in group (64c + 16t) / 32
          const int64_t gi = (static_cast<int64_t>(c) * 64 + 16 * t) >> 5;
          const uint32_t ha = va ? half_scale_bf16x2(__ldg(sa + gi)) : 0u;
          const uint32_t hb = vb ? half_scale_bf16x2(__ldg(sb + gi)) : 0u;
#pragma unroll
          for (int kb = 0; kb < 4; ++kb) {
            const uint32_t a[4] = {bmul2(pair_bits(wa, 2 * kb), ha), bmul2(pair_bits(wb, 2 * kb), hb),
                                   bmul2(pair_bits(wa, 2 * kb + 1), ha),
                                   bmul2(pair_bits(wb, 2 * kb + 1), hb)};
            mma16816(acc0, a, xr[2 * kb], xr[2 * kb + 1]);
            if (kTwoTiles) mma16816(acc1, a, yr[2 * kb], yr[2 * kb + 1]);
          }
        } else {
#pragma unroll
          for (int kb = 0; kb < 4; ++kb) {
            const uint32_t a[4] = {pair_bits(wa, 2 * kb), pair_bits(wb, 2 * kb),
                                   pair_bits(wa, 2 * kb + 1), pair_bits(wb, 2 * kb + 1)};
            mma16816(part0, a, xr[2 * kb], xr[2 * kb + 1]);
            if (kTwoTiles) mma16816(part1, a, yr[2 * kb], yr[2 * kb + 1]);
          }
          if ((c + 1) % chunks_per_group == 0) {
            // close the group: acc += (s / 2) * partial, rows g (slots 0,1) and g+8 (2,3)
            const int64_t gi = (static_cast<int64_t>(c) * 64) >> log2g;
            const float ha = va ? 0.5f * __ldg(sa + gi) : 0.f;
            const float hb = vb ? 0.5f * __ldg(sb + gi) : 0.f;
            acc0[0] = fmaf(ha, part0[0], acc0[0]);
            acc0[1] = fmaf(ha, part0[1], acc0[1]);
            acc0[2] = fmaf(hb, part0[2], acc0[2]);
            acc0[3] = fmaf(hb, part0[3], acc0[3]);
            part0[0] = part0[1] = part0[2] = part0[3] = 0.f;
            if (kTwoTiles) {
              acc1[0] = fmaf(ha, part1[0], acc1[0]);
              acc1[1] = fmaf(ha, part1[1], acc1[1]);
              acc1[2] = fmaf(hb, part1[2], acc1[2]);
              acc1[3] = fmaf(hb, part1[3], acc1[3]);
              part1[0] = part1[1] = part1[2] = part1[3] = 0.f;
            }
          }
        }
      }
    }

    // C fragment: rows g (slots 0, 1) and g + 8 (slots 2, 3), tokens 2t and 2t + 1
    auto store = [&](int token, int64_t row, float v) {
      if (token < m && row < n) {
        if (mat.y_bf16)
          static_cast<__nv_bfloat16*>(mat.y)[token * n + row] = __float2bfloat16_rn(v);
        else
          static_cast<float*>(mat.y)[token * n + row] = v;
      }
    };
    store(2 * t, ra, acc0[0]);
    store(2 * t + 1, ra, acc0[1]);
    store(2 * t, rb, acc0[2]);
    store(2 * t + 1, rb, acc0[3]);
    if (kTwoTiles) {
      store(8 + 2 * t, ra, acc1[0]);
      store(8 + 2 * t + 1, ra, acc1[1]);
      store(8 + 2 * t, rb, acc1[2]);
      store(8 + 2 * t + 1, rb, acc1[3]);
    }
  }
}

}  // namespace

cudaError_t launch_decode(const DecodeBatch& b, int num_sms, cudaStream_t stream) {
  if (b.total_units <= 0) return cudaSuccess;
  const int warps_per_block = kThreads / 32;
  int64_t blocks = (static_cast<int64_t>(b.total_units) + warps_per_block - 1) / warps_per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * 3;
  if (blocks > cap) blocks = cap;
  if (b.m > 8)
    decode_kernel<true><<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(b);
  else
    decode_kernel<false><<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(b);
  return cudaGetLastError();
}

}  // namespace tq
