// dw_gemm.cu — STE weight gradient dW = dY^T X (§3.1: the straight-through
// estimator hands the gradient of the dequantised weight to the latent fp32 W
// unchanged). A plain bf16 x bf16 -> fp32 tcgen05 GEMM; quantisation plays no part.
//
// Output tile: 128 input features k (TMEM lanes) x 256 output features n (TMEM
// columns). The reduction runs over the tokens m, the outer (row) dimension of
// both x [m][k] and dy [m][n], so both operands are MN-major. Each 64-token
// k-block is TMA-loaded as boxes of 64 features x 64 tokens with the 128-byte
// swizzle: two boxes for x (A, 128 features) and four for dy (B, 256 features).
// In the canonical MN-major layout the leading byte offset is the distance between
// 64-feature chunks (one box, 8 KB) and the stride byte offset the distance
// between groups of 8 tokens (1 KB).
//
// Persistent: one CTA per SM walks the tiles, k-tiles fastest, so that the CTAs in
// flight stream the same dy columns. x is loaded with an L2 evict-last policy (it
// is re-read by every n-tile and fits in L2), dy with evict-first. Two TMEM
// accumulators (2 x 256 columns) let the epilogue of one tile overlap the main loop
// of the next. Roles: warp 0 TMA, warp 1 MMA, warps 2-5 epilogue; the epilogue
// thread of lane k writes dW[n][k], so a warp store covers 32 consecutive k of
// one row n (128 contiguous bytes).
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
constexpr int kNumBars = 2 * kStages + 4;
constexpr int kBytes = kBarOff + kNumBars * 8 + 8;
constexpr uint32_t kTmemCols = 512;

__global__ void __launch_bounds__(kThreads, 1)
    dw_gemm_kernel(const __grid_constant__ CUtensorMap tmap_x,
                   const __grid_constant__ CUtensorMap tmap_dy, const DwArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_shared<1024>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nkb = static_cast<int>((args.m + kKBlock - 1) / kKBlock);
  const uint32_t k_tiles = static_cast<uint32_t>((args.k + kDwTileK - 1) / kDwTileK);
  const uint32_t tiles = k_tiles * static_cast<uint32_t>((args.n + kDwTileN - 1) / kDwTileN);
  const int my_tiles =
      blockIdx.x < tiles ? static_cast<int>((tiles - 1 - blockIdx.x) / gridDim.x + 1) : 0;
  const int total = my_tiles * nkb;
  int* status = args.status;
  auto tile_k0 = [&](int i) -> int64_t {
    return static_cast<int64_t>((blockIdx.x + static_cast<uint32_t>(i) * gridDim.x) % k_tiles) * kDwTileK;
  };
  auto tile_n0 = [&](int i) -> int64_t {
    return static_cast<int64_t>((blockIdx.x + static_cast<uint32_t>(i) * gridDim.x) / k_tiles) * kDwTileN;
  };

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_base + kBarOff;
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
  auto accfull_bar = [&](int a) { return bar_base + 8u * (2 * kStages + a); };
  auto accempty_bar = [&](int a) { return bar_base + 8u * (2 * kStages + 2 + a); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kBarOff + kNumBars * 8);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(accfull_bar(a), 1);
      mbar_init(accempty_bar(a), 128);
    }
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
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t keep = policy_evict_last();
      const uint64_t stream = policy_evict_first();
      int issued = 0;
      bool ok = true;
      for (int it = 0; it < total; ++it) {
        const int i = it / nkb, kb = it - i * nkb;
        const int s = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        if (!(ok = mbar_wait(empty_bar(s), ph ^ 1, status))) break;
        const uint32_t a = smem_base + s * kStageBytes;
        const uint32_t b = a + kABytes;
        const int32_t mrow = kb * kKBlock;
        const int64_t k0 = tile_k0(i), n0 = tile_n0(i);
        mbar_arrive_expect_tx(full_bar(s), kStageBytes);
#pragma unroll
        for (int c = 0; c < 2; ++c)
          tma_load_2d_hint(a + c * kBox, &tmap_x, full_bar(s), static_cast<int32_t>(k0 + 64 * c),
                           mrow, keep);
#pragma unroll
        for (int c = 0; c < 4; ++c)
          tma_load_2d_hint(b + c * kBox, &tmap_dy, full_bar(s), static_cast<int32_t>(n0 + 64 * c),
                           mrow, stream);
        ++issued;
      }
      if (!ok) {
        for (int it = issued - 1; it >= 0 && it >= issued - kStages; --it)
          mbar_wait(full_bar(it % kStages), (it / kStages) & 1, status);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(128, kDwTileN, 1, 1);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int acc = i & 1;
        const uint32_t aph = (i >> 1) & 1;
        if (!(ok = mbar_wait(accempty_bar(acc), aph ^ 1, status))) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kDwTileN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!(ok = mbar_wait(full_bar(s), ph, status))) break;
          tc_fence_after();
          const uint32_t a = smem_base + s * kStageBytes;
          const uint32_t b = a + kABytes;
#pragma unroll
          for (int j = 0; j < kKBlock / 16; ++j) {
            // 16 tokens = two 8-token core groups = 2 KB further into each box
            const uint64_t adesc = smem_desc_sw128(a + j * 2048, kBox, 1024);
            const uint64_t bdesc = smem_desc_sw128(b + j * 2048, kBox, 1024);
            mma_ss(d, adesc, bdesc, idesc, (kb | j) != 0);
          }
          mma_commit(empty_bar(s));
        }
        if (ok) mma_commit(accfull_bar(acc));
      }
    }
  } else {
    const int quad = warp & 3;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    for (int i = 0; i < my_tiles; ++i) {
      const int acc = i & 1;
      const uint32_t aph = (i >> 1) & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(accfull_bar(acc), aph, status))) break;
      tc_fence_after();
      const int64_t kk = tile_k0(i) + quad * 32 + lane;
      const int64_t n0 = tile_n0(i);
      const uint32_t d = tmem_base + acc * kDwTileN + lane_off;
#pragma unroll 1
      for (int c = 0; c < kDwTileN; c += 16) {
        uint32_t v[16];
        tmem_ld16(d + c, v);
        tmem_ld_wait16(v);
        if (kk < args.k) {
#pragma unroll
          for (int t = 0; t < 16; ++t) {
            const int64_t n = n0 + c + t;
            if (n < args.n) {
              float* p = args.dw + n * args.k + kk;
              const float val = __uint_as_float(v[t]);
              *p = args.accumulate ? *p + val : val;
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(accempty_bar(acc));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

}  // namespace

size_t dw_smem_bytes() { return kBytes + 1024; }

cudaError_t launch_dw_gemm(const CUtensorMap& tmap_x, const CUtensorMap& tmap_dy,
                           const DwArgs& a, int num_sms, cudaStream_t stream) {
  const size_t smem = dw_smem_bytes();
  cudaError_t e = ensure_smem_limit<dw_gemm_kernel>(static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int64_t tiles = ((a.k + kDwTileK - 1) / kDwTileK) * ((a.n + kDwTileN - 1) / kDwTileN);
  const int64_t grid = tiles < num_sms ? tiles : num_sms;
  dw_gemm_kernel<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(tmap_x, tmap_dy, a);
  return cudaGetLastError();
}

}  // namespace tq
