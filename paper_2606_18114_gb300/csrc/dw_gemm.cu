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
//
// Stream-K tail: the tiles of the whole waves (tiles / grid of them per CTA) go
// round-robin as above; the R = tiles % grid tiles left over are cut into equal
// contiguous runs of k-blocks, one run per CTA, so that every CTA ends at the same
// time instead of R CTAs running one more tile. A tile cut into several pieces has
// each piece's fp32 sum written to the workspace (two slots per CTA: the piece
// that opens its run and the one that closes it); the CTA that completes the last
// piece (a per-tile counter) adds the pieces in k order and writes dW. No CTA
// waits for another. The tail's CTAs read their runs' tokens at different
// offsets, so there dy is kept in L2 (evict-last) like x.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

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
constexpr int kBytes = kBarOff + kNumBars * 8 + 16;  // + TMEM address, "last piece" flag
constexpr uint32_t kTmemCols = 512;
constexpr int kTileFloats = kDwTileK * kDwTileN;

// Stream-K workspace: two tile-sized fp32 slots per CTA, and a completion counter
// per tile of the tail (reset by the CTA that finishes the tile).
__device__ float g_dw_ws[2 * kDwMaxCtas * kTileFloats];
__device__ uint32_t g_dw_cnt[kDwMaxCtas];

// Work of one CTA: its whole tiles (round-robin over the first dp tiles), then
// the pieces of its stream-K run over the rem tail tiles. The tail is cut only
// when it has at least one k-block per CTA (every run then holds a k-block);
// otherwise every tile is whole.
struct DwSched {
  uint32_t grid, dp, rem;  // tiles = dp + rem
  int nkb;                 // k-blocks (64 tokens) per tile
  int64_t units;           // rem * nkb: k-blocks of the tail
  __device__ void init(uint32_t tiles, uint32_t g, int kblocks) {
    grid = g;
    nkb = kblocks;
    rem = tiles % g;
    units = static_cast<int64_t>(rem) * kblocks;
    if (units < g) rem = 0, units = 0;
    dp = tiles - rem;
  }
  __device__ int64_t run_start(uint32_t c) const { return static_cast<int64_t>(c) * units / grid; }
  // CTA whose run holds tail k-block b
  __device__ uint32_t owner(int64_t b) const {
    return static_cast<uint32_t>(((b + 1) * grid - 1) / units);
  }
  __device__ int whole_of(uint32_t c) const { return c < dp ? static_cast<int>((dp - 1 - c) / grid + 1) : 0; }
};

struct DwItem {
  uint32_t tile;
  int kb0, kb1;  // k-blocks [kb0, kb1) of the tile
  int sk;        // -1: a whole-wave tile; else the piece's index within the CTA's run
};

__device__ __forceinline__ int items_of(const DwSched& q, uint32_t c) {
  int n = q.whole_of(c);
  if (q.rem != 0) {
    const int64_t s0 = q.run_start(c), s1 = q.run_start(c + 1);
    if (s1 > s0) n += static_cast<int>((s1 - 1) / q.nkb - s0 / q.nkb + 1);
  }
  return n;
}

__device__ __forceinline__ DwItem item_at(const DwSched& q, uint32_t c, int i) {
  DwItem it;
  const int nw = q.whole_of(c);
  if (i < nw) {
    it.tile = c + static_cast<uint32_t>(i) * q.grid;
    it.kb0 = 0;
    it.kb1 = q.nkb;
    it.sk = -1;
    return it;
  }
  const int j = i - nw;
  const int64_t s0 = q.run_start(c), s1 = q.run_start(c + 1);
  const int64_t r = s0 / q.nkb + j;  // tail tile
  const int64_t b0 = r * q.nkb;
  it.tile = q.dp + static_cast<uint32_t>(r);
  it.kb0 = static_cast<int>((s0 > b0 ? s0 : b0) - b0);
  it.kb1 = static_cast<int>((s1 < b0 + q.nkb ? s1 : b0 + q.nkb) - b0);
  it.sk = j;
  return it;
}

__global__ void __launch_bounds__(kThreads, 1)
    dw_gemm_kernel(const __grid_constant__ CUtensorMap tmap_x,
                   const __grid_constant__ CUtensorMap tmap_dy, const DwArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_shared<1024>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nkb = static_cast<int>((args.m + kKBlock - 1) / kKBlock);
  const uint32_t k_tiles = static_cast<uint32_t>((args.k + kDwTileK - 1) / kDwTileK);
  DwSched q;
  q.init(k_tiles * static_cast<uint32_t>((args.n + kDwTileN - 1) / kDwTileN), gridDim.x, nkb);
  const int my_items = items_of(q, blockIdx.x);
  int* status = args.status;
  auto tile_k0 = [&](uint32_t t) -> int64_t { return static_cast<int64_t>(t % k_tiles) * kDwTileK; };
  auto tile_n0 = [&](uint32_t t) -> int64_t { return static_cast<int64_t>(t / k_tiles) * kDwTileN; };

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_base + kBarOff;
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
  auto accfull_bar = [&](int a) { return bar_base + 8u * (2 * kStages + a); };
  auto accempty_bar = [&](int a) { return bar_base + 8u * (2 * kStages + 2 + a); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kBarOff + kNumBars * 8);
  volatile uint32_t* last_flag = tmem_slot + 1;

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
      for (int i = 0; i < my_items && ok; ++i) {
        const DwItem wi = item_at(q, blockIdx.x, i);
        const int64_t k0 = tile_k0(wi.tile), n0 = tile_n0(wi.tile);
        for (int kb = wi.kb0; kb < wi.kb1; ++kb) {
          const int it = issued;
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!(ok = mbar_wait(empty_bar(s), ph ^ 1, status))) break;
          const uint32_t a = smem_base + s * kStageBytes;
          const uint32_t b = a + kABytes;
          const int32_t mrow = kb * kKBlock;
          mbar_arrive_expect_tx(full_bar(s), kStageBytes);
#pragma unroll
          for (int c = 0; c < 2; ++c)
            tma_load_2d_hint(a + c * kBox, &tmap_x, full_bar(s), static_cast<int32_t>(k0 + 64 * c),
                             mrow, keep);
#pragma unroll
          for (int c = 0; c < 4; ++c)
            tma_load_2d_hint(b + c * kBox, &tmap_dy, full_bar(s), static_cast<int32_t>(n0 + 64 * c),
                             mrow, wi.sk < 0 ? stream : keep);
          ++issued;
        }
      }
      if (!ok) {
        for (int it = issued - 1; it >= 0 && it >= issued - kStages; --it)
          mbar_wait(full_bar(it % kStages), (it / kStages) & 1, status);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, kDwTileN, 1, 1, args.in_f16 != 0);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_items && ok; ++i) {
        const DwItem wi = item_at(q, blockIdx.x, i);
        const int acc = i & 1;
        const uint32_t aph = (i >> 1) & 1;
        if (!(ok = mbar_wait(accempty_bar(acc), aph ^ 1, status))) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kDwTileN;
        for (int kb = wi.kb0; kb < wi.kb1; ++kb, ++it) {
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
            mma_ss(d, adesc, bdesc, idesc, (kb != wi.kb0) || j != 0);
          }
          mma_commit(empty_bar(s));
        }
        if (ok) mma_commit(accfull_bar(acc));
      }
    }
  } else {
    const int quad = warp & 3;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int row = quad * 32 + lane;  // this thread's TMEM lane: feature k0 + row
    // workspace slot of piece j of CTA c's run (its first piece or its last)
    auto slot_of = [&](uint32_t c, int j) -> float* {
      return g_dw_ws + (2 * static_cast<size_t>(c) + (j == 0 ? 0 : 1)) * kTileFloats;
    };
    for (int i = 0; i < my_items; ++i) {
      const DwItem wi = item_at(q, blockIdx.x, i);
      const int acc = i & 1;
      const uint32_t aph = (i >> 1) & 1;
      if (!lanes_wait(accfull_bar(acc), aph, status)) break;
      tc_fence_after();
      const int64_t kk = tile_k0(wi.tile) + row;
      const int64_t n0 = tile_n0(wi.tile);
      const uint32_t d = tmem_base + acc * kDwTileN + lane_off;
      const bool whole = wi.kb0 == 0 && wi.kb1 == nkb;
      if (whole) {
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
        continue;
      }
      // A piece of a tail tile: its sum to this CTA's slot as float4 of four
      // columns, [column / 4][lane] (a warp writes 512 contiguous bytes).
      float4* mine = reinterpret_cast<float4*>(slot_of(blockIdx.x, wi.sk));
#pragma unroll 1
      for (int c = 0; c < kDwTileN; c += 16) {
        uint32_t v[16];
        tmem_ld16(d + c, v);
        tmem_ld_wait16(v);
#pragma unroll
        for (int u = 0; u < 4; ++u)
          mine[(c / 4 + u) * kDwTileK + row] =
              make_float4(__uint_as_float(v[4 * u]), __uint_as_float(v[4 * u + 1]),
                          __uint_as_float(v[4 * u + 2]), __uint_as_float(v[4 * u + 3]));
      }
      // publish the piece; the CTA that completes the tile's last piece reduces it
      const uint32_t r = wi.tile - q.dp;
      const int64_t b0 = static_cast<int64_t>(r) * nkb;
      const uint32_t c_first = q.owner(b0), c_last = q.owner(b0 + nkb - 1);
      const uint32_t pieces = c_last - c_first + 1;
      __threadfence();
      named_bar_sync(1, 128);
      if (row == 0) *last_flag = atomicAdd(&g_dw_cnt[r], 1u) == pieces - 1 ? 1u : 0u;
      named_bar_sync(1, 128);
      if (*last_flag != 0u) {
        __threadfence();
        // the pieces in k order (piece p from CTA c_first + p, in the slot of its
        // first piece when its run starts inside this tile); this CTA's own piece
        // comes from TMEM
        const uint32_t own = blockIdx.x - c_first;
#pragma unroll 1
        for (int c0 = 0; c0 < kDwTileN; c0 += 64) {
          float sum[64];
          for (uint32_t p = 0; p < pieces; ++p) {
            float part[64];
            if (p == own) {
#pragma unroll
              for (int c = 0; c < 64; c += 16) {
                uint32_t v[16];
                tmem_ld16(d + c0 + c, v);
                tmem_ld_wait16(v);
#pragma unroll
                for (int t = 0; t < 16; ++t) part[c + t] = __uint_as_float(v[t]);
              }
            } else {
              const uint32_t pc = c_first + p;
              const float4* src = reinterpret_cast<const float4*>(
                  slot_of(pc, q.run_start(pc) >= b0 ? 0 : 1));
#pragma unroll
              for (int u = 0; u < 16; ++u) {
                const float4 f = __ldcg(src + (c0 / 4 + u) * kDwTileK + row);
                part[4 * u] = f.x;
                part[4 * u + 1] = f.y;
                part[4 * u + 2] = f.z;
                part[4 * u + 3] = f.w;
              }
            }
#pragma unroll
            for (int c = 0; c < 64; ++c) sum[c] = p == 0 ? part[c] : sum[c] + part[c];
          }
          if (kk < args.k) {
#pragma unroll
            for (int c = 0; c < 64; ++c) {
              const int64_t n = n0 + c0 + c;
              if (n < args.n) {
                float* o = args.dw + n * args.k + kk;
                *o = args.accumulate ? *o + sum[c] : sum[c];
              }
            }
          }
        }
        if (row == 0) g_dw_cnt[r] = 0u;  // ready for the next launch
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
  int64_t grid = tiles < num_sms ? tiles : num_sms;
  if (grid > kDwMaxCtas) grid = kDwMaxCtas;
  // The stream-K workspace and counters are shared by the device's dW launches:
  // a launch on another stream than the previous one waits for it.
  static std::mutex mu;
  static cudaEvent_t done[64] = {};
  static cudaStream_t last[64] = {};
  int dev = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (dev < 64) {
    if (done[dev] == nullptr &&
        (e = cudaEventCreateWithFlags(&done[dev], cudaEventDisableTiming)) != cudaSuccess)
      return e;
    if (last[dev] != stream && last[dev] != nullptr &&
        (e = cudaStreamWaitEvent(stream, done[dev], 0)) != cudaSuccess)
      return e;
  }
  dw_gemm_kernel<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(tmap_x, tmap_dy, a);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (dev < 64) {
    if ((e = cudaEventRecord(done[dev], stream)) != cudaSuccess) return e;
    last[dev] = stream;
  }
  return cudaSuccess;
}

}  // namespace tq
