// ts_gemm.cu — W1.58A16 forward and STE dX as tcgen05 GEMMs with the ternary
// weights expanded on chip straight into tensor memory.
//
// Tile: 128 weight rows (TMEM lanes) x BN tokens (TMEM columns), fp32 accumulator
// D^T[row][token] in TMEM. Per 64-wide slice of the reduction ("k-block"):
//   * warp 0 (one lane) TMA-loads the activation tile [BN tokens][64] (128-byte
//     swizzle, K-major B operand) and the packed codes of the slice into one
//     shared-memory stage;
//   * warps 2-5 (one warpgroup; warp w owns TMEM lanes 32*(w%4)..+31) expand the
//     codes of their rows to bf16 pairs bf16(s)*c and tcgen05.st them into the
//     stage's 32 TMEM columns (A operand, K-major, two bf16 per column);
//   * warp 1 (one lane) issues four 128 x BN x 16 tcgen05.mma (A from TMEM, B from
//     shared memory) and commits them to the stage's "empty" barrier.
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

constexpr int kThreads = 192;     // 6 warps: TMA, MMA, 4 x expansion/epilogue
constexpr int kStages = 4;
constexpr int kKBlock = 64;       // reduction elements per stage
constexpr int kCodesBytes = 2048; // codes of one stage: 128 x 16 B (fwd) or 64 x 32 B (dx)

template <int BN>
struct TsLayout {
  static constexpr int kBBytes = BN * kKBlock * 2;             // activation tile
  static constexpr int kStageBytes = ((kBBytes + kCodesBytes + 1023) / 1024) * 1024;
  static constexpr int kScaleOff = kStages * kStageBytes;      // dx: 4 warps x 2 x 64 bf16
  static constexpr int kScaleBytes = 4 * 2 * 64 * 2;
  static constexpr int kBarOff = kScaleOff + kScaleBytes;
  static constexpr int kBarBytes = (3 * kStages + 1) * 8 + 8;
  static constexpr int kBytes = kBarOff + kBarBytes;
  static constexpr int kTxBytes = kBBytes + kCodesBytes;
  static constexpr int kTmemNeed = BN + kStages * 32;
  static constexpr uint32_t kTmemCols = kTmemNeed <= 32 ? 32 : kTmemNeed <= 64 ? 64
                                        : kTmemNeed <= 128 ? 128 : kTmemNeed <= 256 ? 256 : 512;
  static_assert(kTmemNeed <= 512, "tensor memory");
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
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * 128;
  const int64_t m0 = static_cast<int64_t>(blockIdx.y) * BN;
  const int nkb = static_cast<int>((red + kKBlock - 1) / kKBlock);
  int* status = args.status;

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_base + L::kBarOff;
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
  auto afull_bar = [&](int s) { return bar_base + 8u * (2 * kStages + s); };
  const uint32_t acc_bar = bar_base + 8u * (3 * kStages);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kBarOff + (3 * kStages + 1) * 8);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
      mbar_init(afull_bar(s), 128);
    }
    mbar_init(acc_bar, 1);
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
  const uint32_t tmem_acc = tmem_base;
  const uint32_t tmem_a = tmem_base + BN;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1;
        if (!(ok = mbar_wait(empty_bar(s), ph ^ 1, status))) break;
        const uint32_t stage = smem_base + s * L::kStageBytes;
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
        for (int kb = issued - 1; kb >= 0 && kb >= issued - kStages; --kb)
          mbar_wait(full_bar(kb % kStages), (kb / kStages) & 1, status);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(128, BN, 0, 0);
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1;
        if (!mbar_wait(full_bar(s), ph, status)) break;
        if (!mbar_wait(afull_bar(s), ph, status)) break;
        tc_fence_after();
        const uint32_t b_addr = smem_base + s * L::kStageBytes;
#pragma unroll
        for (int j = 0; j < kKBlock / 16; ++j) {
          const uint64_t bdesc = smem_desc_sw128(b_addr + j * 32, 16, 1024);
          mma_ts(tmem_acc, tmem_a + s * 32 + j * 8, bdesc, idesc, (kb | j) != 0);
        }
        mma_commit(empty_bar(s));
      }
      mma_commit(acc_bar);
    }
  } else {
    // ---------------------------------------------------------------- expansion + epilogue
    const int quad = warp & 3;
    const int r_local = quad * 32 + lane;
    const int64_t row = r0 + r_local;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int64_t gpr = args.wk >> args.log2g;  // groups per weight row
    bool ok = true;

    if (MODE == kTsFwd) {
      const float* srow = row < args.wn ? args.scales + row * gpr : nullptr;
      auto load_sc = [&](int kb) -> float2 {
        if (srow == nullptr || kb >= nkb) return make_float2(0.f, 0.f);
        const int64_t gi = (static_cast<int64_t>(kb) * kKBlock) >> args.log2g;
        if (args.log2g == 5) return __ldg(reinterpret_cast<const float2*>(srow + gi));
        const float x = __ldg(srow + gi);
        return make_float2(x, x);
      };
      float2 p0 = load_sc(0), p1 = load_sc(1);
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1;
        const float2 sc = p0;
        p0 = p1;
        p1 = load_sc(kb + 2);
        const bool got = mbar_wait(empty_bar(s), ph ^ 1, status) && mbar_wait(full_bar(s), ph, status);
        if (!(ok = __all_sync(0xffffffffu, got))) break;
        tc_fence_after();
        const uint4 cw = *reinterpret_cast<const uint4*>(smem + s * L::kStageBytes + L::kBBytes +
                                                         r_local * 16);
        const uint32_t hs_lo = half_scale_pair(sc.x, sc.x);
        const uint32_t hs_hi = half_scale_pair(sc.y, sc.y);
        uint32_t a[32];
        expand_word(cw.x, hs_lo, a + 0);
        expand_word(cw.y, hs_lo, a + 8);
        expand_word(cw.z, hs_hi, a + 16);
        expand_word(cw.w, hs_hi, a + 24);
        tmem_st_x32(tmem_a + s * 32 + lane_off, a);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(afull_bar(s));
      }
    } else {
      // dX: this thread is input feature k = row; the warp shares one k-group.
      const int64_t gk = (r0 + quad * 32) >> args.log2g;
      const bool warp_in = (r0 + quad * 32) < args.wk;
      auto load_sc = [&](int kb) -> float2 {
        float2 r = make_float2(0.f, 0.f);
        if (!warp_in || kb >= nkb) return r;
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
      __nv_bfloat16* sbuf = reinterpret_cast<__nv_bfloat16*>(smem + L::kScaleOff) + quad * 128;
      float2 p0 = load_sc(0), p1 = load_sc(1);
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kStages;
        const uint32_t ph = (kb / kStages) & 1;
        const float2 sc = p0;
        p0 = p1;
        p1 = load_sc(kb + 2);
        __nv_bfloat16* sb = sbuf + (kb & 1) * 64;
        sb[lane] = __float2bfloat16_rn(0.5f * sc.x);
        sb[lane + 32] = __float2bfloat16_rn(0.5f * sc.y);
        __syncwarp();
        const bool got = mbar_wait(empty_bar(s), ph ^ 1, status) && mbar_wait(full_bar(s), ph, status);
        if (!(ok = __all_sync(0xffffffffu, got))) break;
        tc_fence_after();
        const uint32_t* tile =
            reinterpret_cast<const uint32_t*>(smem + s * L::kStageBytes + L::kBBytes);
        const uint32_t* spair = reinterpret_cast<const uint32_t*>(sb);
        uint32_t a[32];
#pragma unroll
        for (int p = 0; p < 32; ++p) {
          const uint32_t w0 = tile[(2 * p) * 8 + xw];
          const uint32_t w1 = tile[(2 * p + 1) * 8 + xw];
          const uint32_t t = (__byte_perm(w0, w1, sel) << shift) & 0xC000C000u;
          a[p] = bmul2(t, spair[p]);
        }
        tmem_st_x32(tmem_a + s * 32 + lane_off, a);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(afull_bar(s));
      }
    }

    // ---------------------------------------------------------------- epilogue
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(acc_bar, 0, status));
    tc_fence_after();
    if (ok) {
      const int64_t m = args.m;
      if (BN == 16) {
        uint32_t v[32] = {};
        tmem_ld_x16(tmem_acc + lane_off, v);
        tmem_ld_wait(v);
        if (row < rows) {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (m0 + i < m) store_out(args.out, (m0 + i) * rows + row, __uint_as_float(v[i]),
                                      args.out_bf16);
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t v[32];
          tmem_ld_x32(tmem_acc + lane_off + c, v);
          tmem_ld_wait(v);
          if (row < rows) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (m0 + c + i < m)
                store_out(args.out, (m0 + c + i) * rows + row, __uint_as_float(v[i]),
                          args.out_bf16);
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
    tmem_dealloc(tmem_base, L::kTmemCols);
  }
}

template <int MODE, int BN>
cudaError_t launch_impl(const CUtensorMap& tb, const CUtensorMap& tc, const TsArgs& a,
                        cudaStream_t stream) {
  using L = TsLayout<BN>;
  // at least ~100 KB per CTA keeps residency to at most two CTAs per SM, so the
  // tensor-memory allocations (<= 256 columns each when two fit) never wait
  size_t smem = L::kBytes + 1024;
  if (L::kTmemCols > 256) smem = smem < 120 * 1024 ? 120 * 1024 : smem;
  else smem = smem < 100 * 1024 ? 100 * 1024 : smem;
  auto kern = ts_gemm_kernel<MODE, BN>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int64_t rows = MODE == kTsFwd ? a.wn : a.wk;
  dim3 grid(static_cast<unsigned>((rows + 127) / 128), static_cast<unsigned>((a.m + BN - 1) / BN));
  kern<<<grid, kThreads, smem, stream>>>(tb, tc, a);
  return cudaGetLastError();
}

}  // namespace

int ts_tile_tokens(int64_t m) { return m <= 16 ? 16 : 256; }

size_t ts_smem_bytes(int bn) {
  return bn == 16 ? TsLayout<16>::kBytes : TsLayout<256>::kBytes;
}

cudaError_t launch_ts_gemm(int mode, int bn, const CUtensorMap& tb, const CUtensorMap& tc,
                           const TsArgs& a, cudaStream_t stream) {
  if (mode == kTsFwd) {
    if (bn == 16) return launch_impl<kTsFwd, 16>(tb, tc, a, stream);
    if (bn == 256) return launch_impl<kTsFwd, 256>(tb, tc, a, stream);
  } else {
    if (bn == 16) return launch_impl<kTsDx, 16>(tb, tc, a, stream);
    if (bn == 256) return launch_impl<kTsDx, 256>(tb, tc, a, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace tq
