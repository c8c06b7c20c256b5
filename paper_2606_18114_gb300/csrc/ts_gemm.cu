// ts_gemm.cu — W1.58A16 forward and STE dX as persistent tcgen05 GEMMs with the
// ternary weights expanded on chip straight into tensor memory.
//
// Output tile: 128 weight rows (TMEM lanes) x BN tokens (TMEM columns), fp32
// accumulator D^T[row][token] in TMEM. One CTA per SM walks the tiles
// (rows fastest, so the CTAs in flight share the activation tile in L2). Per
// 128-wide slice of the reduction ("k-block"):
//   * warp 0 (one lane) TMA-loads the activation tile [BN tokens][128] (two
//     64-wide boxes with the 128-byte swizzle, K-major B operand) and the packed
//     codes of the slice into one shared-memory stage;
//   * warps 6-13, two warpgroups each covering half of the slice (warp w owns
//     TMEM lanes 32*(w%4)..+31), expand the codes of their rows to bf16 pairs
//     bf16(s)*c as soon as the codes land, and tcgen05.st them into the A stage
//     (K-major, two bf16 per column) once the MMAs that last read it are done;
//   * warp 1 (one lane) issues eight 128 x BN x 16 tcgen05.mma (A from TMEM, B
//     from shared memory) and one commit, which frees the smem stage and, later,
//     the A stage;
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
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace tq {
namespace {

constexpr int kEpiWarp0 = 2;                 // warps 2..5: epilogue warpgroup
constexpr int kExpWarp0 = 6;                 // warps 6..13: two expansion warpgroups
constexpr int kThreads = 14 * 32;
constexpr int kKBlock = 128;                 // reduction elements per stage
constexpr int kCodesBytes = 4096;            // 128 rows x 8 code words
// dX with at most this many k-blocks per tile (n <= 4096) runs the ping-pong layout
constexpr int kDxPingPongMaxKb = 32;

// Rings: kSmem shared-memory stages (activation tile as two 64-wide swizzled halves
// + codes, filled by TMA) and kAStages tensor-memory stages of expanded weights
// (64 columns = 128 k each). Each stage's MMAs are committed to the smem stage's
// "empty" barrier (refill by TMA); when the smem ring is at least as deep as the
// A ring, that same commit tells the expansion, kAStages iterations later, that
// the A stage is free, otherwise a second commit goes to the A stage's barrier.
// Tensor memory (512 columns) holds kAcc accumulators of BN columns plus the A ring:
//   forward, 256 tokens ("ping-pong"): the two halves of tensor memory, 256
//     columns each, swap roles every tile. Tile i accumulates in half i % 2 while
//     its A ring (four stages of 64 columns, stage kb % 4 for k-block kb of the
//     tile) lives in the other half; tile i + 1's A ring is tile i's accumulator.
//     The epilogue drains tile i in four 64-column chunks and releases each chunk
//     ("drained") as soon as it is in registers, before storing it; the expansion
//     fills stage c of tile i + 1 once chunk c is released. The MMAs of the next
//     tile so restart after a quarter of the drain instead of all of it (an fp32
//     tile leaves the SM at ~30 B per cycle, a quarter of the tile's MMA time):
//     in_proj forward 0.385 -> 0.379 ms alone, 0.382 -> 0.373 in the step, less
//     than the drain's share because the stores then compete with the activation
//     stream (~66 B per cycle into each SM) instead of pausing it. A deep A ring
//     hides the commit -> expansion -> MMA round trip: two A stages beside a ring of
//     three 128-token accumulator halves ran the forward in 0.411 ms;
//   dX, 256 tokens: with more than kDxPingPongMaxKb k-blocks per tile, one
//     accumulator and four A stages in a ring over the launch (its tiles are 67
//     k-blocks long at in_proj, so the drain is a small share: the ping-pong layout
//     ran it 1.6 % slower); with fewer, ping-pong as the forward (out_proj, 16
//     k-blocks: 0.210 -> 0.201 ms; equal at 32 and 48);
//   16 tokens: two accumulators and four A stages.
template <int MODE, int BN, bool PP>
struct TsLayout {
  static_assert(BN == 16 || BN == 256, "tile tokens");
  static_assert(!PP || BN == 256, "ping-pong: two 256-column halves");
  static constexpr bool kPingPong = PP;
  static constexpr int kSmem = BN == 16 ? 16 : 3;
  static constexpr int kAStages = 4;
  static constexpr int kAcc = BN == 256 ? 1 : 2;
  static_assert(!kPingPong || (kAcc * BN == 256 && kAStages * 64 == 256), "two halves");
  static constexpr bool kReleaseViaSmem = kSmem >= kAStages;
  static constexpr int kSubBytes = BN * 64 * 2;                // one 64-wide k half
  static constexpr int kBBytes = 2 * kSubBytes;
  static constexpr int kStageBytes = ((kBBytes + kCodesBytes + 1023) / 1024) * 1024;
  static constexpr int kScaleOff = kSmem * kStageBytes;     // dx: 2 WG x 4 warps x 2 x 64 bf16
  static constexpr int kScaleBytes = 2 * 4 * 2 * 64 * 2;
  static constexpr int kBarOff = kScaleOff + kScaleBytes;
  static constexpr int kNumBars = 2 * kSmem + 2 * kAStages + 2 * kAcc + 4;  // + drained
  static constexpr int kBytes = kBarOff + kNumBars * 8 + 8;
  static constexpr int kTxBytes = kBBytes + kCodesBytes;
  static constexpr int kTmemNeed = kAcc * BN + kAStages * 64;
  static constexpr uint32_t kTmemCols = kTmemNeed <= 32 ? 32 : kTmemNeed <= 64 ? 64
                                        : kTmemNeed <= 128 ? 128 : kTmemNeed <= 256 ? 256 : 512;
  static_assert(kTmemNeed <= 512, "tensor memory");
  static_assert(BN % 16 == 0, "epilogue chunks");
};

// Two 16-bit products in the activation type (bf16, or fp16 with F16).
template <bool F16>
__device__ __forceinline__ uint32_t bmul2(uint32_t a, uint32_t b) {
  uint32_t d;
  if constexpr (F16)
    asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  else
    asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// s / 2 rounded to the activation type, as its 16 bits.
template <bool F16>
__device__ __forceinline__ uint16_t half_scale_bits(float s) {
  if constexpr (F16)
    return __half_as_ushort(__float2half_rn(0.5f * s));
  else
    return __bfloat16_as_ushort(__float2bfloat16_rn(0.5f * s));
}

template <bool F16>
__device__ __forceinline__ uint32_t half_scale_pair(float lo, float hi) {
  // round(s)/2 in both halves; s/2 is exact in fp32 and rounding commutes with it.
  return static_cast<uint32_t>(half_scale_bits<F16>(lo)) |
         (static_cast<uint32_t>(half_scale_bits<F16>(hi)) << 16);
}

// 16 codes of one word -> 8 A-operand columns of two 16-bit values, times the
// scale pair (the codes expand to +-2 = 0x4000 / 0xC000 in bf16 and fp16 alike).
template <bool F16>
__device__ __forceinline__ void expand_word(uint32_t w, uint32_t hs, uint32_t* a) {
#pragma unroll
  for (int j = 0; j < 8; ++j) a[j] = bmul2<F16>((w << (14 - 2 * j)) & 0xC000C000u, hs);
}

template <int MODE, int BN, bool F16, bool PP>
__global__ void __launch_bounds__(kThreads, 1)
    ts_gemm_kernel(const __grid_constant__ CUtensorMap tmap_b,
                   const __grid_constant__ CUtensorMap tmap_codes, const TsArgs args) {
  using L = TsLayout<MODE, BN, PP>;
  constexpr int kSmem = L::kSmem, kAS = L::kAStages, kAcc = L::kAcc;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_shared<1024>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t rows = MODE == kTsFwd ? args.wn : args.wk;
  const int64_t red = MODE == kTsFwd ? args.wk : args.wn;
  const int nkb = static_cast<int>((red + kKBlock - 1) / kKBlock);
  // tile t = blockIdx.x + i * gridDim.x covers rows (t % row_tiles) * 128 and
  // tokens (t / row_tiles) * BN; tile counts fit in 32 bits (checked on the host)
  const uint32_t row_tiles = static_cast<uint32_t>((rows + 127) / 128);
  const uint32_t tiles = row_tiles * static_cast<uint32_t>((args.m + BN - 1) / BN);
  const int my_tiles =
      blockIdx.x < tiles ? static_cast<int>((tiles - 1 - blockIdx.x) / gridDim.x + 1) : 0;
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
  auto empty_bar = [&](int s) { return bar_base + 8u * (kSmem + s); };
  auto afull_bar = [&](int a) { return bar_base + 8u * (2 * kSmem + a); };
  auto aempty_bar = [&](int a) { return bar_base + 8u * (2 * kSmem + kAS + a); };
  auto accfull_bar = [&](int a) { return bar_base + 8u * (2 * kSmem + 2 * kAS + a); };
  auto accempty_bar = [&](int a) { return bar_base + 8u * (2 * kSmem + 2 * kAS + kAcc + a); };
  // ping-pong: chunk c (64 columns) of the last tile's accumulator is in registers
  auto drained_bar = [&](int c) { return bar_base + 8u * (2 * kSmem + 2 * kAS + 2 * kAcc + c); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kBarOff + L::kNumBars * 8);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kSmem; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < kAS; ++a) {
      mbar_init(afull_bar(a), 8);  // one arrival per expansion warp
      mbar_init(aempty_bar(a), 1);
    }
    for (int a = 0; a < kAcc; ++a) {
      mbar_init(accfull_bar(a), 1);
      mbar_init(accempty_bar(a), 4);  // one arrival per epilogue warp
    }
    for (int c = 0; c < 4; ++c) mbar_init(drained_bar(c), 4);  // one per epilogue warp
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
  const uint32_t tmem_a = tmem_base + kAcc * BN;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int it = 0; it < total; ++it) {
        const int i = it / nkb, kb = it - i * nkb;
        const int s = it % kSmem;
        const uint32_t ph = (it / kSmem) & 1;
        if (!(ok = mbar_wait(empty_bar(s), ph ^ 1, status))) break;
        const uint32_t stage = smem_base + s * L::kStageBytes;
        const int64_t r0 = tile_r0(i), m0 = tile_m0(i);
        mbar_arrive_expect_tx(full_bar(s), L::kTxBytes);
        tma_load_2d(stage, &tmap_b, full_bar(s), kb * kKBlock, static_cast<int32_t>(m0));
        tma_load_2d(stage + L::kSubBytes, &tmap_b, full_bar(s), kb * kKBlock + 64,
                    static_cast<int32_t>(m0));
        if (MODE != kTsDx)  // codes (forward) or codes_t (dX): rows = this tile's rows
          tma_load_2d(stage + L::kBBytes, &tmap_codes, full_bar(s), kb * (kKBlock / 16),
                      static_cast<int32_t>(r0));
        else
          tma_load_2d(stage + L::kBBytes, &tmap_codes, full_bar(s),
                      static_cast<int32_t>(r0 / 16), kb * kKBlock);
        ++issued;
      }
      if (!ok) {  // let copies already in flight land before the CTA winds down
        for (int it = issued - 1; it >= 0 && it >= issued - kSmem; --it)
          mbar_wait(full_bar(it % kSmem), (it / kSmem) & 1, status);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (L::kPingPong && lane == 0) {
      // No wait for the accumulator: the first MMA of tile i + 1 waits for its A
      // stage, which the expansion fills only after the epilogue has taken chunk 0
      // of tile i, i.e. after every MMA of tile i completed (both halves are free).
      constexpr uint32_t idesc = idesc_bf16(128, BN, 0, 0, F16);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const uint32_t d = tmem_base + 256u * (i & 1);
        const uint32_t a0 = tmem_base + 256u * ((i + 1) & 1);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kSmem, as = kb % kAS;
          const int use = i * ((nkb - as + kAS - 1) / kAS) + kb / kAS;  // of stage as
          // afull implies full: the expansion warps waited on this stage's TMA
          // barrier before they arrived, so one wait orders both operands.
          if (!(ok = mbar_wait(afull_bar(as), use & 1, status))) break;
          tc_fence_after();
          const uint32_t b_addr = smem_base + s * L::kStageBytes;
#pragma unroll
          for (int j = 0; j < kKBlock / 16; ++j) {
            const uint64_t bdesc =
                smem_desc_sw128(b_addr + (j >> 2) * L::kSubBytes + (j & 3) * 32, 16, 1024);
            mma_ts(d, a0 + as * 64 + j * 8, bdesc, idesc, (kb | j) != 0);
          }
          mma_commit(empty_bar(s));
          mma_commit(aempty_bar(as));
        }
        if (ok) mma_commit(accfull_bar(0));
      }
    } else if (!L::kPingPong && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(128, BN, 0, 0, F16);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int acc = i % kAcc;
        const uint32_t aph = (i / kAcc) & 1;
        if (!(ok = mbar_wait(accempty_bar(acc), aph ^ 1, status))) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * BN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kSmem, as = it % kAS;
          // afull implies full: the expansion warps waited on this stage's TMA
          // barrier before they arrived, so one wait orders both operands.
          if (!(ok = mbar_wait(afull_bar(as), (it / kAS) & 1, status))) break;
          tc_fence_after();
          const uint32_t b_addr = smem_base + s * L::kStageBytes;
#pragma unroll
          for (int j = 0; j < kKBlock / 16; ++j) {
            const uint64_t bdesc =
                smem_desc_sw128(b_addr + (j >> 2) * L::kSubBytes + (j & 3) * 32, 16, 1024);
            mma_ts(d, tmem_a + as * 64 + j * 8, bdesc, idesc, (kb | j) != 0);
          }
          mma_commit(empty_bar(s));
          if (!L::kReleaseViaSmem) mma_commit(aempty_bar(as));
        }
        if (ok) mma_commit(accfull_bar(acc));
      }
    }
  } else if (warp < kExpWarp0) {
    // ---------------------------------------------------------------- epilogue
    const int quad = warp & 3;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int64_t m = args.m;
    if constexpr (L::kPingPong) {
      for (int i = 0; i < my_tiles; ++i) {
        if (!lanes_wait(accfull_bar(0), i & 1, status)) break;
        tc_fence_after();
        const int64_t row = tile_r0(i) + quad * 32 + lane;
        const int64_t m0 = tile_m0(i);
        const uint32_t d = tmem_base + 256u * (i & 1) + lane_off;
        const int mvalid = static_cast<int>(m - m0 < BN ? m - m0 : BN);
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t v[4][16];
#pragma unroll
          for (int q = 0; q < 4; ++q) tmem_ld16(d + 64 * c + 16 * q, v[q]);
          tmem_ld_wait16(v[0]);
          tmem_regs_ready16(v[1]);
          tmem_regs_ready16(v[2]);
          tmem_regs_ready16(v[3]);
          // the chunk is in registers: its columns become an A stage of the next tile
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(drained_bar(c));
          if (row < rows) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int cc = 64 * c + 16 * q;
              if (args.out_bf16) {
                __nv_bfloat16* p = static_cast<__nv_bfloat16*>(args.out) + (m0 + cc) * rows + row;
#pragma unroll
                for (int t = 0; t < 16; ++t, p += rows)
                  if (cc + t < mvalid) *p = __float2bfloat16_rn(__uint_as_float(v[q][t]));
              } else {
                float* p = static_cast<float*>(args.out) + (m0 + cc) * rows + row;
#pragma unroll
                for (int t = 0; t < 16; ++t, p += rows)
                  if (cc + t < mvalid) *p = __uint_as_float(v[q][t]);
              }
            }
          }
        }
      }
    } else {
    for (int i = 0; i < my_tiles; ++i) {
      const int acc = i % kAcc;
      const uint32_t aph = (i / kAcc) & 1;
      if (!lanes_wait(accfull_bar(acc), aph, status)) break;
      tc_fence_after();
      const int64_t row = tile_r0(i) + quad * 32 + lane;
      const int64_t m0 = tile_m0(i);
      const uint32_t d = tmem_base + acc * BN + lane_off;
      // element (m0 + c + t, row) of out; tokens beyond m are not stored
      const int mvalid = static_cast<int>(m - m0 < BN ? m - m0 : BN);
      // four 16-column loads in flight per wait
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 64) {
        uint32_t v[4][16];
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_ld16(d + c0 + 16 * q, v[q]);
        tmem_ld_wait16(v[0]);
        tmem_regs_ready16(v[1]);
        tmem_regs_ready16(v[2]);
        tmem_regs_ready16(v[3]);
        if (row < rows) {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int c = c0 + 16 * q;
            if (args.out_bf16) {
              __nv_bfloat16* p = static_cast<__nv_bfloat16*>(args.out) + (m0 + c) * rows + row;
#pragma unroll
              for (int t = 0; t < 16; ++t, p += rows)
                if (c + t < mvalid) *p = __float2bfloat16_rn(__uint_as_float(v[q][t]));
            } else {
              float* p = static_cast<float*>(args.out) + (m0 + c) * rows + row;
#pragma unroll
              for (int t = 0; t < 16; ++t, p += rows)
                if (c + t < mvalid) *p = __uint_as_float(v[q][t]);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(accempty_bar(acc));
    }
    }
  } else {
    // ---------------------------------------------------------------- expansion
    // Both warpgroups take every k-block: warpgroup wg fills A columns
    // [32 wg, 32 wg + 32) of the stage, i.e. reduction offsets [64 wg, 64 wg + 64).
    const int wg = (warp - kExpWarp0) >> 2;
    const int quad = warp & 3;
    const int r_local = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int64_t gpr = args.wk >> args.log2g;  // groups per weight row

    // Cursor over k-blocks: tile i, k-block kb, first row of the tile.
    struct Cursor {
      int it, i, kb;
      int64_t r0;
    };
    auto cursor_at = [&](int it) {
      Cursor c;
      c.it = it;
      c.i = it / nkb;
      c.kb = it - c.i * nkb;
      c.r0 = tile_r0(c.i);
      return c;
    };
    auto advance = [&](Cursor& c) {
      ++c.it;
      if (++c.kb == nkb) {
        c.kb = 0;
        ++c.i;
        c.r0 = tile_r0(c.i);
      }
    };
    // A stage of a k-block: it % kAS in a ring over the whole launch, or (ping-pong)
    // kb % kAS in the half of tensor memory that is not the tile's accumulator.
    auto stage_of = [&](const Cursor& c) { return L::kPingPong ? c.kb % kAS : c.it % kAS; };
    auto stage_col = [&](const Cursor& c) -> uint32_t {
      if constexpr (L::kPingPong)
        return tmem_base + 256u * ((c.i + 1) & 1) + (c.kb % kAS) * 64;
      else
        return tmem_a + (c.it % kAS) * 64;
    };
    // The A stage is free once the MMAs that last read it are done: those of
    // iteration it - kAS; ping-pong: those of k-block kb - kAS of the tile, or, for
    // the tile's first use of the stage, the epilogue has taken the previous tile's
    // accumulator chunk kb (those columns).
    auto a_free = [&](const Cursor& c) -> bool {
      if constexpr (L::kPingPong) {
        const int as = c.kb % kAS;
        if (c.kb < kAS) return c.i == 0 || lanes_wait(drained_bar(as), (c.i - 1) & 1, status);
        const int use = c.i * ((nkb - as + kAS - 1) / kAS) + c.kb / kAS;  // of stage as
        return lanes_wait(aempty_bar(as), (use - 1) & 1, status);
      } else {
        const int it = c.it;
        if (L::kReleaseViaSmem) {
          if (it < kAS) return true;
          const int j = it - kAS;
          return lanes_wait(empty_bar(j % kSmem), (j / kSmem) & 1, status);
        }
        return lanes_wait(aempty_bar(it % kAS), ((it / kAS) & 1) ^ 1, status);
      }
    };
    auto publish = [&](const Cursor& c, const uint32_t* a) {
      const uint32_t col = stage_col(c) + wg * 32 + lane_off;
      tc_fence_after();
      tmem_st_x16(col, a);
      tmem_st_x16(col + 16, a + 16);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(afull_bar(stage_of(c)));
    };
    Cursor cur = cursor_at(0);
    Cursor pre = cursor_at(2);

    if (MODE == kTsFwd) {
      auto load_sc = [&](const Cursor& c) -> float2 {
        const int64_t row = c.r0 + r_local;
        if (c.it >= total || row >= args.wn) return make_float2(0.f, 0.f);
        const float* srow = args.scales + row * gpr;
        const int64_t gi = (static_cast<int64_t>(c.kb) * kKBlock + wg * 64) >> args.log2g;
        if (args.log2g == 5) return __ldg(reinterpret_cast<const float2*>(srow + gi));
        const float x = __ldg(srow + gi);
        return make_float2(x, x);
      };
      float2 p0 = load_sc(cur), p1 = load_sc(cursor_at(1));
      for (; cur.it < total; advance(cur), advance(pre)) {
        const int it = cur.it;
        const int s = it % kSmem;
        const float2 sc = p0;
        p0 = p1;
        p1 = load_sc(pre);
        // Expand as soon as the codes have landed; only the tensor-memory store
        // waits for the A stage.
        if (!lanes_wait(full_bar(s), (it / kSmem) & 1, status)) break;
        const uint4 cw = *reinterpret_cast<const uint4*>(smem + s * L::kStageBytes + L::kBBytes +
                                                         r_local * 32 + wg * 16);
        const uint32_t hs_lo = half_scale_pair<F16>(sc.x, sc.x);
        const uint32_t hs_hi = half_scale_pair<F16>(sc.y, sc.y);
        uint32_t a[32];
        expand_word<F16>(cw.x, hs_lo, a + 0);
        expand_word<F16>(cw.y, hs_lo, a + 8);
        expand_word<F16>(cw.z, hs_hi, a + 16);
        expand_word<F16>(cw.w, hs_hi, a + 24);
        if (!a_free(cur)) break;
        publish(cur, a);
      }
    } else {
      // dX: this thread is input feature k = row; a warp shares one k-group, and
      // warpgroup wg covers rows n in [kb*128 + 64 wg, kb*128 + 64 wg + 64). The
      // scale varies along n: each warp stages the bf16(s)/2 of its 64 rows n in
      // shared memory and reads them as pairs.
      auto load_sc = [&](const Cursor& c) -> float2 {
        float2 r = make_float2(0.f, 0.f);
        const int64_t kwarp = c.r0 + quad * 32;
        if (c.it >= total || kwarp >= args.wk) return r;
        const int64_t gk = kwarp >> args.log2g;
        const int64_t n_a = static_cast<int64_t>(c.kb) * kKBlock + wg * 64 + lane;
        const int64_t n_b = n_a + 32;
        if (n_a < args.wn) r.x = __ldg(args.scales + n_a * gpr + gk);
        if (n_b < args.wn) r.y = __ldg(args.scales + n_b * gpr + gk);
        return r;
      };
      uint16_t* sbuf = reinterpret_cast<uint16_t*>(smem + L::kScaleOff) + (wg * 4 + quad) * 128;
      float2 p0 = load_sc(cur), p1 = load_sc(cursor_at(1));
      if (MODE == kTsDxT) {
        // codes_t: this thread's row k of the transposed codes holds rows n along it,
        // so the expansion is the forward's with a scale pair per pair of rows n.
        for (; cur.it < total; advance(cur), advance(pre)) {
          const int it = cur.it;
          const int s = it % kSmem;
          const float2 sc = p0;
          p0 = p1;
          p1 = load_sc(pre);
          uint16_t* sb = sbuf + (it & 1) * 64;
          sb[lane] = half_scale_bits<F16>(sc.x);
          sb[lane + 32] = half_scale_bits<F16>(sc.y);
          __syncwarp();
          if (!lanes_wait(full_bar(s), (it / kSmem) & 1, status)) break;
          const uint4 cw = *reinterpret_cast<const uint4*>(smem + s * L::kStageBytes + L::kBBytes +
                                                           r_local * 32 + wg * 16);
          const uint4* sp = reinterpret_cast<const uint4*>(sb);  // 32 pairs of rows n
          const uint32_t words[4] = {cw.x, cw.y, cw.z, cw.w};
          uint32_t a[32];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint4 s0 = sp[2 * q], s1 = sp[2 * q + 1];
            const uint32_t pr[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
#pragma unroll
            for (int j = 0; j < 8; ++j)
              a[8 * q + j] = bmul2<F16>((words[q] << (14 - 2 * j)) & 0xC000C000u, pr[j]);
          }
          if (!a_free(cur)) break;
          publish(cur, a);
        }
      } else {
      // this thread's 2-bit field inside a code word of its 16-wide k slice
      const int i16 = r_local & 15;
      const int pos = 16 * (i16 & 1) + 2 * (i16 >> 1);
      const uint32_t sel = static_cast<uint32_t>(((pos >> 3) << 4) | ((4 + (pos >> 3)) << 12));
      const int shift = 6 - (pos & 7);
      const int xw = r_local >> 4;
      for (; cur.it < total; advance(cur), advance(pre)) {
        const int it = cur.it;
        const int s = it % kSmem;
        const float2 sc = p0;
        p0 = p1;
        p1 = load_sc(pre);
        uint16_t* sb = sbuf + (it & 1) * 64;
        sb[lane] = half_scale_bits<F16>(sc.x);
        sb[lane + 32] = half_scale_bits<F16>(sc.y);
        __syncwarp();
        if (!lanes_wait(full_bar(s), (it / kSmem) & 1, status)) break;
        const uint32_t* tile =
            reinterpret_cast<const uint32_t*>(smem + s * L::kStageBytes + L::kBBytes) + wg * 64 * 8;
        const uint32_t* spair = reinterpret_cast<const uint32_t*>(sb);
        uint32_t a[32];
#pragma unroll
        for (int p = 0; p < 32; ++p) {
          const uint32_t w0 = tile[(2 * p) * 8 + xw];
          const uint32_t w1 = tile[(2 * p + 1) * 8 + xw];
          const uint32_t t = (__byte_perm(w0, w1, sel) << shift) & 0xC000C000u;
          a[p] = bmul2<F16>(t, spair[p]);
        }
        if (!a_free(cur)) break;
        publish(cur, a);
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

template <int MODE, int BN, bool F16, bool PP>
cudaError_t launch_impl(const CUtensorMap& tb, const CUtensorMap& tc, const TsArgs& a,
                        int num_sms, cudaStream_t stream) {
  using L = TsLayout<MODE, BN, PP>;
  // Enough shared memory that two CTAs never share an SM (each holds up to 512
  // tensor-memory columns).
  size_t smem = L::kBytes + 1024;
  if (smem < 116 * 1024) smem = 116 * 1024;
  auto kern = ts_gemm_kernel<MODE, BN, F16, PP>;
  cudaError_t e = ensure_smem_limit<ts_gemm_kernel<MODE, BN, F16, PP>>(static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int64_t rows = MODE == kTsFwd ? a.wn : a.wk;
  const int64_t tiles = ((rows + 127) / 128) * ((a.m + BN - 1) / BN);
  const int64_t grid = tiles < num_sms ? tiles : num_sms;
  kern<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(tb, tc, a);
  return cudaGetLastError();
}

}  // namespace

int ts_tile_tokens(int mode, int64_t m) { return m <= 16 ? 16 : 256; }

namespace {
template <bool F16>
cudaError_t launch_typed(int mode, int bn, const CUtensorMap& tb, const CUtensorMap& tc,
                         const TsArgs& a, int num_sms, cudaStream_t stream) {
  // dX tiles reduce over n: with few k-blocks per tile the drain of the single
  // accumulator is a large share of each tile, so short reductions take ping-pong
  const bool dx_pp = (a.wn + kKBlock - 1) / kKBlock <= kDxPingPongMaxKb;
  if (mode == kTsFwd) {
    if (bn == 256) return launch_impl<kTsFwd, 256, F16, true>(tb, tc, a, num_sms, stream);
  } else if (mode == kTsDx) {
    if (bn == 16) return launch_impl<kTsDx, 16, F16, false>(tb, tc, a, num_sms, stream);
    if (bn == 256)
      return dx_pp ? launch_impl<kTsDx, 256, F16, true>(tb, tc, a, num_sms, stream)
                   : launch_impl<kTsDx, 256, F16, false>(tb, tc, a, num_sms, stream);
  } else if (mode == kTsDxT) {
    if (bn == 16) return launch_impl<kTsDxT, 16, F16, false>(tb, tc, a, num_sms, stream);
    if (bn == 256)
      return dx_pp ? launch_impl<kTsDxT, 256, F16, true>(tb, tc, a, num_sms, stream)
                   : launch_impl<kTsDxT, 256, F16, false>(tb, tc, a, num_sms, stream);
  }
  return cudaErrorInvalidValue;
}
}  // namespace

cudaError_t launch_ts_gemm(int mode, int bn, const CUtensorMap& tb, const CUtensorMap& tc,
                           const TsArgs& a, int num_sms, cudaStream_t stream) {
  return a.in_f16 ? launch_typed<true>(mode, bn, tb, tc, a, num_sms, stream)
                  : launch_typed<false>(mode, bn, tb, tc, a, num_sms, stream);
}

}  // namespace tq
