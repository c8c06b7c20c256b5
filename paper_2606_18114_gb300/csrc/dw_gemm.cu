// dw_gemm.cu — STE weight gradient dW = dY^T X (§3.1: the straight-through
// estimator hands the gradient of the dequantised weight to the latent fp32 W
// unchanged). A plain bf16 x bf16 -> fp32 tcgen05 GEMM; quantisation plays no part.
//
// Tile: 128 input features k (TMEM lanes) x 256 output features n (TMEM columns);
// the reduction runs over the tokens m, which is the outer (row) dimension of both
// x [m][k] and dy [m][n], so both operands are MN-major. Each 64-token k-block
// is TMA-loaded as boxes of 64 features x 64 tokens with the 128-byte swizzle:
// two boxes for x (A, 128 features) and four for dy (B, 256 features). In the
// canonical MN-major layout the leading byte offset is the distance between
// 64-feature chunks (one box, 8 KB) and the stride byte offset the distance
// between groups of 8 tokens (1 KB).
//
// The epilogue thread of lane k writes dW[n][k] for the tile's columns n, so a
// warp's store covers 32 consecutive k of one row n (128 contiguous bytes).
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace tq {
namespace {

constexpr int kThreads = 192;  // TMA, MMA, 4 epilogue warps
constexpr int kStages = 4;
constexpr int kKBlock = 64;    // tokens per stage
constexpr int kBox = 64 * 64 * 2;
constexpr int kABytes = 2 * kBox;   // 128 features
constexpr int kBBytes = 4 * kBox;   // 256 features
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kBarOff = kStages * kStageBytes;
constexpr int kBytes = kBarOff + (2 * kStages + 1) * 8 + 8;
constexpr uint32_t kTmemCols = 256;

__global__ void __launch_bounds__(kThreads, 1)
    dw_gemm_kernel(const __grid_constant__ CUtensorMap tmap_x,
                   const __grid_constant__ CUtensorMap tmap_dy, const DwArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t k0 = static_cast<int64_t>(blockIdx.x) * kDwTileK;
  const int64_t n0 = static_cast<int64_t>(blockIdx.y) * kDwTileN;
  const int nkb = static_cast<int>((args.m + kKBlock - 1) / kKBlock);
  int* status = args.status;

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_base + kBarOff;
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
  const uint32_t acc_bar = bar_base + 8u * (2 * kStages);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kBarOff + (2 * kStages + 1) * 8);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_bar, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmap_x);
    tma_prefetch_desc(&tmap_dy);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_acc = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1;
        if (!(ok = mbar_wait(empty_bar(s), ph ^ 1, status))) break;
        const uint32_t a = smem_base + s * kStageBytes;
        const uint32_t b = a + kABytes;
        const int32_t mrow = kb * kKBlock;
        mbar_arrive_expect_tx(full_bar(s), kStageBytes);
#pragma unroll
        for (int c = 0; c < 2; ++c)
          tma_load_2d(a + c * kBox, &tmap_x, full_bar(s), static_cast<int32_t>(k0 + 64 * c), mrow);
#pragma unroll
        for (int c = 0; c < 4; ++c)
          tma_load_2d(b + c * kBox, &tmap_dy, full_bar(s), static_cast<int32_t>(n0 + 64 * c), mrow);
        ++issued;
      }
      if (!ok) {
        for (int kb = issued - 1; kb >= 0 && kb >= issued - kStages; --kb)
          mbar_wait(full_bar(kb % kStages), (kb / kStages) & 1, status);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(128, kDwTileN, 1, 1);
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1;
        if (!mbar_wait(full_bar(s), ph, status)) break;
        tc_fence_after();
        const uint32_t a = smem_base + s * kStageBytes;
        const uint32_t b = a + kABytes;
#pragma unroll
        for (int j = 0; j < kKBlock / 16; ++j) {
          // 16 tokens = two 8-token core groups = 2 KB further into each box
          const uint64_t adesc = smem_desc_sw128(a + j * 2048, kBox, 1024);
          const uint64_t bdesc = smem_desc_sw128(b + j * 2048, kBox, 1024);
          mma_ss(tmem_acc, adesc, bdesc, idesc, (kb | j) != 0);
        }
        mma_commit(empty_bar(s));
      }
      mma_commit(acc_bar);
    }
  } else {
    const int quad = warp & 3;
    const int64_t kk = k0 + quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const bool ok = __all_sync(0xffffffffu, mbar_wait(acc_bar, 0, status));
    tc_fence_after();
    if (ok) {
#pragma unroll 1
      for (int c = 0; c < kDwTileN; c += 32) {
        uint32_t v[32];
        tmem_ld_x32(tmem_acc + lane_off + c, v);
        tmem_ld_wait(v);
        if (kk < args.k) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int64_t n = n0 + c + i;
            if (n < args.n) {
              float* p = args.dw + n * args.k + kk;
              const float val = __uint_as_float(v[i]);
              *p = args.accumulate ? *p + val : val;
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_acc, kTmemCols);
  }
}

}  // namespace

size_t dw_smem_bytes() { return kBytes + 1024; }

cudaError_t launch_dw_gemm(const CUtensorMap& tmap_x, const CUtensorMap& tmap_dy,
                           const DwArgs& a, cudaStream_t stream) {
  const size_t smem = dw_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(dw_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(static_cast<unsigned>((a.k + kDwTileK - 1) / kDwTileK),
            static_cast<unsigned>((a.n + kDwTileN - 1) / kDwTileN));
  dw_gemm_kernel<<<grid, kThreads, smem, stream>>>(tmap_x, tmap_dy, a);
  return cudaGetLastError();
}

}  // namespace tq
