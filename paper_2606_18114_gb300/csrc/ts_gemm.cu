// ts_gemm.cu — W1.58A16 forward and STE dX as persistent tcgen05 GEMMs with the
// ternary weights expanded on chip straight into tensor memory.
//
// Output tile: 128 weight rows (TMEM lanes) x BN tokens (TMEM columns), fp32
// accumulator D^T[row][token] in TMEM, two accumulators so that the epilogue of
// one tile overlaps the main loop of the next. One CTA per SM walks the tiles
// (rows fastest, so the CTAs in flight share the activation tile in L2). Per
// 64-wide slice of the reduction ("k-block"):
//   * warp 0 (one lane) TMA-loads the activation tile [BN tokens][64] (128-byte
//     swizzle, K-major B operand) and the packed codes of the slice into one
//     shared-memory stage;
//   * warps 6-13, two warpgroups taking alternate k-blocks (warp w owns TMEM
//     lanes 32*(w%4)..+31), expand the codes of their rows to bf16 pairs
//     bf16(s)*c and tcgen05.st them into the stage's 32 TMEM columns (A operand,
//     K-major, two bf16 per column);
//   * warp 1 (one lane) issues four 128 x BN x 16 tcgen05.mma (A from TMEM, B
//     from shared memory) and commits them to the stage's "empty" barrier;
//   * warps 2-5 (one warpgroup) drain the finished accumulator with tcgen05.ld
//     and store it; each warp store covers 32 consecutive rows of one token.
// The expanded weights never touch shared memory, so shared-memory bandwidth is
// spent only on the activation tile (TMA write + MMA read).
//
// Expansion: with the packed layout of include/tq.h, pair j of a code word
// becomes the bf16x2 (2*c_2j, 2*c_2j+1) by ((w << (14 - 2j)) & 0xC000C000); one
// bf16x2 multiply by bf16(s)/2 gives (bf16(s)*c_2j, bf16(s)*c_2j+1) exactly.
//
// Forward (§3.1): rows are output features n, the reduction runs over k, the
// scale is per row and k-group. dX (STE, §3.1): rows are input features k, the
// reduction runs over n, the scale varies along the reduction (per n), and each
// thread picks its own 2-bit field out of the codes of 64 consecutive rows n.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace tq {
namespace {

constexpr int kEpiWarp0 = 2;                 // warps 2..5: epilogue warpgroup
constexpr int kExpWarp0 = 6;                 // warps 6..13: two expansion warpgroups
constexpr int kThreads = 14 * 32;
constexpr int kStages = 4;
constexpr int kKBlock = 64;                  // reduction elements per stage
constexpr int kCodesBytes = 2048;            // 128 x 16 B (fwd) or 64 x 32 B (dx)

template <int BN>
struct TsLayout {
  static constexpr int kBBytes = BN * kKBlock * 2;
  static constexpr int kStageBytes = ((kBBytes + kCodesBytes + 1023) / 1024) * 1024;
  static constexpr int kScaleOff = kStages * kStageBytes;   // dx: 2 WG x 4 warps x 2 x 64 bf16
  static constexpr int kScaleBytes = 2 * 4 * 2 * 64 * 2;
  static constexpr int kBarOff = kScaleOff + kScaleBytes;
  static constexpr int kNumBars = 3 * kStages + 4;
  static constexpr int kBytes = kBarOff + kNumBars * 8 + 8;
  static constexpr int kTxBytes = kBBytes + kCodesBytes;
  static constexpr int kTmemNeed = 2 * BN + kStages * 32;
  static constexpr uint32_t kTmemCols = kTmemNeed <= 32 ? 32 : kTmemNeed <= 64 ? 64
                                        : kTmemNeed <= 128 ? 128 : kTmemNeed <= 256 ? 256 : 512;
  static_assert(kTmemNeed <= 512, "tensor memory");
  static_assert(BN % 32 == 0 || BN == 16, "epilogue chunks");
};

__device__ __forceinline__ uint32_t bmul2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

__device__ __forceinline__ uint32_t half_scale_pair(float lo, float hi) {
  // bf16(s)/2 in both halves; s/2 is exact in fp32 and rounding commutes with it.
  const __nv_bfloat16 l = __float2bfloat16_rn(0.5f * lo);
  const __nv_bfloat16 h = __float2bfloat16_rn(0.5f * hi);
  return static_cast<uint32_t>(__bfloat16_as_ushort(l)) |
         (static_cast<uint32_t>(__bfloat16_as_ushort(h)) << 16);
}

// 16 codes of one word -> 8 bf16x2 A-operand columns, times the scale pair.
__device__ __forceinline__ void expand_word(uint32_t w, uint32_t hs, uint32_t* a) {
#pragma unroll
  for (int j = 0; j < 8; ++j) a[j] = bmul2((w << (14 - 2 * j)) & 0xC000C000u, hs);
}

__device__ __forceinline__ void store_out(void* out, int64_t idx, float v, int bf16) {
  if (bf16)
    static_cast<__nv_bfloat16*>(out)[idx] = __float2bfloat16_rn(v);
  else
    static_cast<float*>(out)[idx] = v;
}

template <int MODE, int BN>
__global__ void __launch_bounds__(kThreads, 1)
    ts_gemm_kernel(const __grid_constant__ CUtensorMap tmap_b,
                   const __grid_constant__ CUtensorMap tmap_codes, const TsArgs args) {
  using L = TsLayout<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t rows = MODE == kTsFwd ? args.wn : args.wk;
  const int64_t red = MODE == kTsFwd ? args.wk : args.wn;
  const int nkb = static_cast<int>((red + kKBlock - 1) / kKBlock);
  // tile t = blockIdx.x + i * gridDim.x covers rows (t % row_tiles) * 128 and
  // tokens (t / row_tiles) * BN; tile counts fit in 32 bits (checked on the host)
  const uint32_t row_tiles = static_cast<uint32_t>((rows + 127) / 128);
  const uint32_t tiles = row_tiles * static_cast<uint32_t>((args.m + BN - 1) / BN);
  const int my_tiles = blockIdx.x < tiles ? static_cast<int>((tiles - 1 - blockIdx.x) / gridDim.x + 1) : 0;
  const int total = my_tiles * nkb;  // k-blocks this CTA runs
  int* status = args.status;
  auto tile_r0 = [&](int i) -> int64_t {
    return static_cast<int64_t>((blockIdx.x + static_cast<uint32_t>(i) * gridDim.x) % row_tiles) * 128;
  };
  auto tile_m0 = [&](int i) -> int64_t {
    return static_cast<int64_t>((blockIdx.x + static_cast<uint32_t>(i) * gridDim.x) / row_tiles) * BN;
  };

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_base + L::kBarOff;
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
  auto afull_bar = [&](int s) { return bar_base + 8u * (2 * kStages + s); };
  auto accfull_bar = [&](int a) { return bar_base + 8u * (3 * kStages + a); };
  auto accempty_bar = [&](int a) { return bar_base + 8u * (3 * kStages + 2 + a); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kBarOff + L::kNumBars * 8);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
      mbar_init(afull_bar(s), 128);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(accfull_bar(a), 1);
      mbar_init(accempty_bar(a), 128);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), L::kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmap_b);
    tma_prefetch_desc(&tmap_codes);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t tmem_a = tmem_base + 2 * BN;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int it = 0; it < total; ++it) {
        const int i = it / nkb, kb = it - i * nkb;
        const int s = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        if (!(ok = mbar_wait(empty_bar(s), ph ^ 1, status))) break;
        const uint32_t stage = smem_base + s * L::kStageBytes;
        const int64_t r0 = tile_r0(i), m0 = tile_m0(i);
        mbar_arrive_expect_tx(full_bar(s), L::kTxBytes);
        tma_load_2d(stage, &tmap_b, full_bar(s), kb * kKBlock, static_cast<int32_t>(m0));
        if (MODE == kTsFwd)
          tma_load_2d(stage + L::kBBytes, &tmap_codes, full_bar(s), kb * (kKBlock / 16),
                      static_cast<int32_t>(r0));
        else
          tma_load_2d(stage + L::kBBytes, &tmap_codes, full_bar(s),
                      static_cast<int32_t>(r0 / 16), kb * kKBlock);
        ++issued;
      }
      if (!ok) {  // let copies already in flight land before the CTA winds down
        for (int it = issued - 1; it >= 0 && it >= issued - kStages; --it)
          mbar_wait(full_bar(it % kStages), (it / kStages) & 1, status);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(128, BN, 0, 0);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int acc = i & 1;
        const uint32_t aph = (i >> 1) & 1;
        if (!(ok = mbar_wait(accempty_bar(acc), aph ^ 1, status))) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * BN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!(ok = mbar_wait(full_bar(s), ph, status) && mbar_wait(afull_bar(s), ph, status)))
            break;
          tc_fence_after();
          const uint32_t b_addr = smem_base + s * L::kStageBytes;
#pragma unroll
          for (int j = 0; j < kKBlock / 16; ++j) {
            const uint64_t bdesc = smem_desc_sw128(b_addr + j * 32, 16, 1024);
            mma_ts(d, tmem_a + s * 32 + j * 8, bdesc, idesc, (kb | j) != 0);
          }
          mma_commit(empty_bar(s));
        }
        if (ok) mma_commit(accfull_bar(acc));
      }
    }
  } else if (warp < kExpWarp0) {
    // ---------------------------------------------------------------- epilogue
    const int quad = warp & 3;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int64_t m = args.m;
    for (int i = 0; i < my_tiles; ++i) {
      const int acc = i & 1;
      const uint32_t aph = (i >> 1) & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(accfull_bar(acc), aph, status))) break;
      tc_fence_after();
      const int64_t row = tile_r0(i) + quad * 32 + lane;
      const int64_t m0 = tile_m0(i);
      const uint32_t d = tmem_base + acc * BN + lane_off;
      if (BN == 16) {
        uint32_t v[32] = {};
        tmem_ld_x16(d, v);
        tmem_ld_wait(v);
        if (row < rows) {
#pragma unroll
          for (int t = 0; t < 16; ++t)
            if (m0 + t < m)
              store_out(args.out, (m0 + t) * rows + row, __uint_as_float(v[t]), args.out_bf16);
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          uint32_t v[16];
          tmem_ld16(d + c, v);
          tmem_ld_wait16(v);
          if (row < rows) {
#pragma unroll
            for (int t = 0; t < 16; ++t)
              if (m0 + c + t < m)
                store_out(args.out, (m0 + c + t) * rows + row, __uint_as_float(v[t]),
                          args.out_bf16);
          }
        }
      }
      tc_fence_before();
      mbar_arrive(accempty_bar(acc));
    }
  } else {
    // ---------------------------------------------------------------- expansion
    const int wg = (warp - kExpWarp0) >> 2;   // 0 or 1: takes k-blocks it % 2 == wg
    const int quad = warp & 3;
    const int r_local = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int64_t gpr = args.wk >> args.log2g;  // groups per weight row

    if (MODE == kTsFwd) {
      auto load_sc = [&](int it) -> float2 {
        if (it >= total) return make_float2(0.f, 0.f);
        const int i = it / nkb, kb = it - i * nkb;
        const int64_t row = tile_r0(i) + r_local;
        if (row >= args.wn) return make_float2(0.f, 0.f);
        const float* srow = args.scales + row * gpr;
        const int64_t gi = (static_cast<int64_t>(kb) * kKBlock) >> args.log2g;
        if (args.log2g == 5) return __ldg(reinterpret_cast<const float2*>(srow + gi));
        const float x = __ldg(srow + gi);
        return make_float2(x, x);
      };
      float2 p0 = load_sc(wg), p1 = load_sc(wg + 2);
      for (int it = wg; it < total; it += 2) {
        const int s = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        const float2 sc = p0;
        p0 = p1;
        p1 = load_sc(it + 4);
        const bool got = mbar_wait(empty_bar(s), ph ^ 1, status) && mbar_wait(full_bar(s), ph, status);
        if (!__all_sync(0xffffffffu, got)) break;
        tc_fence_after();
        const uint4 cw = *reinterpret_cast<const uint4*>(smem + s * L::kStageBytes + L::kBBytes +
                                                         r_local * 16);
        const uint32_t hs_lo = half_scale_pair(sc.x, sc.x);
        const uint32_t hs_hi = half_scale_pair(sc.y, sc.y);
        uint32_t a[16];
        expand_word(cw.x, hs_lo, a + 0);
        expand_word(cw.y, hs_lo, a + 8);
        tmem_st_x16(tmem_a + s * 32 + lane_off, a);
        expand_word(cw.z, hs_hi, a + 0);
        expand_word(cw.w, hs_hi, a + 8);
        tmem_st_x16(tmem_a + s * 32 + 16 + lane_off, a);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(afull_bar(s));
      }
    } else {
      // dX: this thread is input feature k = row; a warp shares one k-group.
      auto load_sc = [&](int it) -> float2 {
        float2 r = make_float2(0.f, 0.f);
        if (it >= total) return r;
        const int i = it / nkb, kb = it - i * nkb;
        const int64_t kwarp = tile_r0(i) + quad * 32;
        if (kwarp >= args.wk) return r;
        const int64_t gk = kwarp >> args.log2g;
        const int64_t n_a = static_cast<int64_t>(kb) * kKBlock + lane;
        const int64_t n_b = n_a + 32;
        if (n_a < args.wn) r.x = __ldg(args.scales + n_a * gpr + gk);
        if (n_b < args.wn) r.y = __ldg(args.scales + n_b * gpr + gk);
        return r;
      };
      // this thread's 2-bit field inside a code word of its 16-wide k slice
      const int i16 = r_local & 15;
      const int pos = 16 * (i16 & 1) + 2 * (i16 >> 1);
      const uint32_t sel = static_cast<uint32_t>(((pos >> 3) << 4) | ((4 + (pos >> 3)) << 12));
      const int shift = 6 - (pos & 7);
      const int xw = r_local >> 4;
      __nv_bfloat16* sbuf =
          reinterpret_cast<__nv_bfloat16*>(smem + L::kScaleOff) + (wg * 4 + quad) * 128;
      float2 p0 = load_sc(wg), p1 = load_sc(wg + 2);
      int local = 0;
      for (int it = wg; it < total; it += 2, ++local) {
        const int s = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        const float2 sc = p0;
        p0 = p1;
        p1 = load_sc(it + 4);
        __nv_bfloat16* sb = sbuf + (local & 1) * 64;
        sb[lane] = __float2bfloat16_rn(0.5f * sc.x);
        sb[lane + 32] = __float2bfloat16_rn(0.5f * sc.y);
        __syncwarp();
        const bool got = mbar_wait(empty_bar(s), ph ^ 1, status) && mbar_wait(full_bar(s), ph, status);
        if (!__all_sync(0xffffffffu, got)) break;
        tc_fence_after();
        const uint32_t* tile =
            reinterpret_cast<const uint32_t*>(smem + s * L::kStageBytes + L::kBBytes);
        const uint32_t* spair = reinterpret_cast<const uint32_t*>(sb);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint32_t a[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int p = 16 * h + q;
            const uint32_t w0 = tile[(2 * p) * 8 + xw];
            const uint32_t w1 = tile[(2 * p + 1) * 8 + xw];
            const uint32_t t = (__byte_perm(w0, w1, sel) << shift) & 0xC000C000u;
            a[q] = bmul2(t, spair[p]);
          }
          tmem_st_x16(tmem_a + s * 32 + 16 * h + lane_off, a);
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(afull_bar(s));
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, L::kTmemCols);
  }
}

template <int MODE, int BN>
cudaError_t launch_impl(const CUtensorMap& tb, const CUtensorMap& tc, const TsArgs& a,
                        int num_sms, cudaStream_t stream) {
  using L = TsLayout<BN>;
  // Enough shared memory that two CTAs never share an SM (each holds up to 512
  // tensor-memory columns).
  size_t smem = L::kBytes + 1024;
  if (smem < 116 * 1024) smem = 116 * 1024;
  auto kern = ts_gemm_kernel<MODE, BN>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int64_t rows = MODE == kTsFwd ? a.wn : a.wk;
  const int64_t tiles = ((rows + 127) / 128) * ((a.m + BN - 1) / BN);
  const int64_t grid = tiles < num_sms ? tiles : num_sms;
  kern<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(tb, tc, a);
  return cudaGetLastError();
}

}  // namespace

int ts_tile_tokens(int64_t m) { return m <= 16 ? 16 : 192; }

cudaError_t launch_ts_gemm(int mode, int bn, const CUtensorMap& tb, const CUtensorMap& tc,
                           const TsArgs& a, int num_sms, cudaStream_t stream) {
  if (mode == kTsFwd) {
    if (bn == 16) return launch_impl<kTsFwd, 16>(tb, tc, a, num_sms, stream);
    if (bn == 192) return launch_impl<kTsFwd, 192>(tb, tc, a, num_sms, stream);
  } else {
    if (bn == 16) return launch_impl<kTsDx, 16>(tb, tc, a, num_sms, stream);
    if (bn == 192) return launch_impl<kTsDx, 192>(tb, tc, a, num_sms, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace tq
