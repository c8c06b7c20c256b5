// dw_gemm.cu — STE weight gradient dW = dY^T X (§3.1: the straight-through
// estimator hands the gradient of the dequantised weight to the latent fp32 W
// unchanged). A plain bf16 x bf16 -> fp32 tcgen05 GEMM; quantisation plays no part.
//
// CTA pairs: a cluster of two CTAs on two SMs computes a 256 x 256 tile (input
// features k x output features n) with cta_group::2 MMAs issued by the leader
// (rank 0): CTA r loads rows k0 + 128 r .. + 127 of the A operand (x) and columns
// n0 + 128 r .. + 127 of the B operand (dy) into its own shared memory, the pair's
// M = 256 MMA reads both halves of both operands, and CTA r's tensor memory holds
// D for its 128 features k (TMEM lanes) x all 256 output features (columns). Each
// SM thus feeds the tensor cores 32 KB of operands per 64 tokens instead of the
// 48 KB a single CTA's 128 x 256 tile reads, which is what capped the one-SM form.
//
// The reduction runs over the tokens m, the outer (row) dimension of both x [m][k]
// and dy [m][n], so both operands are MN-major. Each 128-token k-block is
// TMA-loaded as boxes of 64 features x 64 tokens with the 128-byte swizzle (four for
// x, four for dy per CTA; 128-token stages halve the hand-offs per flop of 64-token
// ones: in_proj 0.352 -> 0.346 ms). In the canonical MN-major layout the leading byte offset is the
// distance between 64-feature chunks (one box, 8 KB) and the stride byte offset the
// distance between groups of 8 tokens (1 KB).
//
// Hand-offs. Each CTA's producer waits on its own "empty" barrier and loads into its
// own "full" barrier; the peer's idle MMA warp relays the completion of each of its
// stages to the leader ("peer full", a plain remote arrive: the bytes are in the
// peer's shared memory once its phase completes), so the leader's MMA thread issues
// a stage once both halves have landed. The leader's commits are multicast to both
// CTAs: "empty" (the stage may be refilled), "accumulator full" (each epilogue
// drains its own TMEM). Both CTAs' epilogue warps arrive on the leader's
// "accumulator empty" (with release: their TMEM reads precede the next MMAs). The
// single threads on the pipeline's path (producers, MMA issuer, relay) spin on their
// barriers: a suspended waiter resumed late after an arrival from the other SM.
//
// Persistent: the pairs walk the tiles, k-tiles fastest, so that the pairs in
// flight stream the same dy columns: a wave of 76 pair tiles covers all eight
// k-tiles of in_proj (x, 67 MB) and 9.5 n-tiles of dy. Both operands are loaded
// with an L2 evict-last hint (the same DRAM bytes as no hint; dy evict-first read
// 26 % more and ran 8 % slower: the eight pairs of an n-tile drift apart in token).
// Whole tiles alternate their token direction (see item_at), so a wave starts on
// the x blocks the previous one read last. Two TMEM
// accumulators (2 x 256 columns) let the epilogue of one tile overlap the main loop
// of the next. Roles: warp 0 TMA, warp 1 MMA (leader) or relay (peer), warps 2-5
// epilogue; the epilogue thread of lane k writes dW[n][k], so a warp store covers
// 32 consecutive k of one row n (128 contiguous bytes).
//
// Stream-K tail: the tiles of the whole waves (tiles / pairs of them per pair) go
// round-robin as above; the R = tiles % pairs tiles left over are cut into equal
// contiguous runs of k-blocks, one run per pair, so that every pair ends at the
// same time instead of R pairs running one more tile. A tile cut into several
// pieces has each CTA's half of each piece written to the workspace (two slots per
// CTA: the piece that opens its run and the one that closes it); for each half, the
// CTA that completes the last piece (a per-tile, per-half counter) adds the pieces
// in k order and writes dW. No CTA waits for another pair.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "kernels.cuh"
#include "ptx.cuh"

namespace tq {
namespace {

constexpr int kThreads = 192;  // TMA, MMA / relay, 4 epilogue warps
constexpr int kStages = 3;
constexpr int kKBlock = 128;   // tokens per stage
constexpr int kBox = 64 * 64 * 2;
constexpr int kABytes = 4 * kBox;   // this CTA's 128 features k, two 64-token blocks
constexpr int kBBytes = 4 * kBox;   // this CTA's 128 output features n, two 64-token blocks
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kBarOff = kStages * kStageBytes;
constexpr int kNumBars = 3 * kStages + 4;  // full, empty, peer full; 2 acc full, 2 acc empty
constexpr int kBytes = kBarOff + kNumBars * 8 + 16;  // + TMEM address, "last piece" flag
constexpr uint32_t kTmemCols = 512;
constexpr int kTileFloats = kDwTileK * kDwTileN;  // one CTA's half of a pair tile

// Stream-K workspace: two half-tile fp32 slots per CTA, and a completion counter
// per half of each tile of the tail (reset by the CTA that finishes it).
__device__ float g_dw_ws[2 * kDwMaxCtas * kTileFloats];
__device__ uint32_t g_dw_cnt[kDwMaxCtas];

// Work of one pair: its whole tiles (round-robin over the first dp tiles), then
// the pieces of its stream-K run over the rem tail tiles. The tail is cut only
// when it has at least one k-block per pair (every run then holds a k-block);
// otherwise every tile is whole.
struct DwSched {
  uint32_t grid, dp, rem;  // grid: pairs; tiles = dp + rem
  int nkb;                 // k-blocks (128 tokens) per tile
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
  // pair whose run holds tail k-block b
  __device__ uint32_t owner(int64_t b) const {
    return static_cast<uint32_t>(((b + 1) * grid - 1) / units);
  }
  __device__ int whole_of(uint32_t c) const { return c < dp ? static_cast<int>((dp - 1 - c) / grid + 1) : 0; }
};

struct DwItem {
  uint32_t tile;
  int kb0, kb1;  // k-blocks [kb0, kb1) of the tile
  int sk;        // -1: a whole-wave tile; else the piece's index within the pair's run
  bool rev;      // the k-blocks are loaded last to first
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
    // Whole tiles alternate their token direction, the last one running down to
    // token 0 where the tail's pieces start: each wave begins on the x blocks that
    // the wave before read last, which L2 still holds.
    it.tile = c + static_cast<uint32_t>(i) * q.grid;
    it.kb0 = 0;
    it.kb1 = q.nkb;
    it.sk = -1;
    it.rev = ((nw - 1 - i) & 1) == 0;
    return it;
  }
  // A run that crosses into the next tile takes that tile's first k-blocks before
  // the end of the tile it starts in. Every pair then works at token offset
  // tau + d at time tau, d in [0, nkb - run length] (0 for those first pieces, the
  // run's start for a run inside one tile, nkb - run length for the ends), so the
  // pairs sharing an x or dy block reach it within that window rather than up to a
  // whole tile apart (in_proj, 44 tail tiles: 867 -> 598 MB of DRAM reads per
  // launch). The piece keeps its index (0: the piece that opens the run) whatever
  // the order.
  const int64_t s0 = q.run_start(c), s1 = q.run_start(c + 1);
  const int two = (s1 - 1) / q.nkb != s0 / q.nkb;
  const int j = two ? 1 - (i - nw) : i - nw;
  const int64_t r = s0 / q.nkb + j;  // tail tile
  const int64_t b0 = r * q.nkb;
  it.tile = q.dp + static_cast<uint32_t>(r);
  it.kb0 = static_cast<int>((s0 > b0 ? s0 : b0) - b0);
  it.kb1 = static_cast<int>((s1 < b0 + q.nkb ? s1 : b0 + q.nkb) - b0);
  it.sk = j;
  it.rev = false;
  return it;
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    dw_gemm_kernel(const __grid_constant__ CUtensorMap tmap_x,
                   const __grid_constant__ CUtensorMap tmap_dy, const DwArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_shared<1024>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const uint32_t pair = blockIdx.x >> 1;
  const int nkb = static_cast<int>((args.m + kKBlock - 1) / kKBlock);
  const uint32_t k_tiles = static_cast<uint32_t>((args.k + kDwPairK - 1) / kDwPairK);
  DwSched q;
  q.init(k_tiles * static_cast<uint32_t>((args.n + kDwTileN - 1) / kDwTileN), gridDim.x >> 1, nkb);
  const int my_items = items_of(q, pair);
  int* status = args.status;
  // this CTA's first feature k of tile t, and the tile's first output feature n
  auto tile_k0 = [&](uint32_t t) -> int64_t {
    return static_cast<int64_t>(t % k_tiles) * kDwPairK + kDwTileK * rank;
  };
  auto tile_n0 = [&](uint32_t t) -> int64_t { return static_cast<int64_t>(t / k_tiles) * kDwTileN; };

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_base + kBarOff;
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
  auto pfull_bar = [&](int s) { return bar_base + 8u * (2 * kStages + s); };
  auto accfull_bar = [&](int a) { return bar_base + 8u * (3 * kStages + a); };
  auto accempty_bar = [&](int a) { return bar_base + 8u * (3 * kStages + 2 + a); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kBarOff + kNumBars * 8);
  volatile uint32_t* last_flag = tmem_slot + 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
      mbar_init(pfull_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(accfull_bar(a), 1);
      mbar_init(accempty_bar(a), 8);  // the four epilogue warps of each CTA
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish_pair();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmap_x);
    tma_prefetch_desc(&tmap_dy);
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers are initialised before either signals the other
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      const uint64_t keep = policy_evict_last();
      int issued = 0;
      bool ok = true;
      for (int i = 0; i < my_items && ok; ++i) {
        const DwItem wi = item_at(q, pair, i);
        const int64_t k0 = tile_k0(wi.tile), n0 = tile_n0(wi.tile) + kDwTileK * rank;
        for (int kb = wi.kb0; kb < wi.kb1; ++kb) {
          const int it = issued;
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!(ok = mbar_wait_spin(empty_bar(s), ph ^ 1, status))) break;
          const uint32_t a = smem_base + s * kStageBytes;
          const uint32_t b = a + kABytes;
          const int32_t mrow = (wi.rev ? wi.kb0 + wi.kb1 - 1 - kb : kb) * kKBlock;
          mbar_arrive_expect_tx(full_bar(s), kStageBytes);
#pragma unroll
          for (int c = 0; c < 4; ++c)  // box c: features 64 (c & 1), tokens 64 (c >> 1)
            tma_load_2d_hint(a + c * kBox, &tmap_x, full_bar(s), static_cast<int32_t>(k0 + 64 * (c & 1)),
                             mrow + 64 * (c >> 1), keep);
#pragma unroll
          for (int c = 0; c < 4; ++c)
            tma_load_2d_hint(b + c * kBox, &tmap_dy, full_bar(s), static_cast<int32_t>(n0 + 64 * (c & 1)),
                             mrow + 64 * (c >> 1), keep);
          ++issued;
        }
      }
      if (!ok) {  // nothing may still write this CTA's ring when it exits
        for (int it = issued - 1; it >= 0 && it >= issued - kStages; --it)
          mbar_wait_spin(full_bar(it % kStages), (it / kStages) & 1, status);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank != 0) {
      // ---------------------------------------------------------------- relay (peer)
      // Tell the leader when each of this CTA's stages has landed.
      const uint32_t leader_pfull0 = map_to_rank(pfull_bar(0), 0);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_items && ok; ++i) {
        const DwItem wi = item_at(q, pair, i);
        for (int kb = wi.kb0; kb < wi.kb1; ++kb, ++it) {
          const int s = it % kStages;
          if (!(ok = mbar_wait_spin(full_bar(s), (it / kStages) & 1, status))) break;
          mbar_arrive_remote_signal(leader_pfull0 + 8u * s);
        }
      }
    } else if (lane == 0) {
      // ---------------------------------------------------------------- MMA (leader)
      const uint32_t idesc = idesc_bf16(2 * kDwTileK, kDwTileN, 1, 1, args.in_f16 != 0);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_items && ok; ++i) {
        const DwItem wi = item_at(q, pair, i);
        const int acc = i & 1;
        const uint32_t aph = (i >> 1) & 1;
        if (!(ok = mbar_wait_spin(accempty_bar(acc), aph ^ 1, status))) break;
        tc_fence_after();
        const uint32_t d = tmem_base + acc * kDwTileN;
        for (int kb = wi.kb0; kb < wi.kb1; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!(ok = mbar_wait_spin(full_bar(s), ph, status) && mbar_wait_spin(pfull_bar(s), ph, status))) break;
          tc_fence_after();
          const uint32_t a = smem_base + s * kStageBytes;
          const uint32_t b = a + kABytes;
#pragma unroll
          for (int j = 0; j < kKBlock / 16; ++j) {
            // 16 tokens = two 8-token core groups = 2 KB further into each box; the
            // second 64-token block starts two boxes further
            const uint64_t adesc = smem_desc_sw128(a + (j >> 2) * 2 * kBox + (j & 3) * 2048, kBox, 1024);
            const uint64_t bdesc = smem_desc_sw128(b + (j >> 2) * 2 * kBox + (j & 3) * 2048, kBox, 1024);
            mma_ss_pair(d, adesc, bdesc, idesc, (kb != wi.kb0) || j != 0);
          }
          mma_commit_pair(empty_bar(s));
        }
        if (ok) mma_commit_pair(accfull_bar(acc));
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int quad = warp & 3;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int row = quad * 32 + lane;  // this thread's TMEM lane: feature k0 + row
    const uint32_t leader_accempty0 = map_to_rank(accempty_bar(0), 0);
    // timeout tests only: the leader's first epilogue warp of pair 0 withholds its
    // first "accumulator empty" arrival
    bool withhold = pair == 0 && rank == 0 && warp == 2 && test_withhold(status, kWithholdDwAccEmpty);
    auto release = [&](int acc) {  // this warp is done with the accumulator
      tc_fence_before();
      __syncwarp();
      if (lane == 0 && !withhold) mbar_arrive_remote(leader_accempty0 + 8u * acc);
      withhold = false;
    };
    // workspace slot of piece j of the run of pair c (its first piece or its last),
    // for this CTA's half
    auto slot_of = [&](uint32_t c, int j) -> float* {
      return g_dw_ws + (2 * static_cast<size_t>(2 * c + rank) + (j == 0 ? 0 : 1)) * kTileFloats;
    };
    for (int i = 0; i < my_items; ++i) {
      const DwItem wi = item_at(q, pair, i);
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
        release(acc);
        continue;
      }
      // A piece of a tail tile: this CTA's half of its sum to this CTA's slot as
      // float4 of four columns, [column / 4][lane] (a warp writes 512 contiguous bytes).
      float4* mine = reinterpret_cast<float4*>(slot_of(pair, wi.sk));
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
      // publish the piece; for each half, the CTA that completes the tile's last
      // piece reduces it
      const uint32_t r = wi.tile - q.dp;
      const int64_t b0 = static_cast<int64_t>(r) * nkb;
      const uint32_t c_first = q.owner(b0), c_last = q.owner(b0 + nkb - 1);
      const uint32_t pieces = c_last - c_first + 1;
      uint32_t* cnt = &g_dw_cnt[2 * r + rank];
      __threadfence();
      named_bar_sync(1, 128);
      if (row == 0) *last_flag = atomicAdd(cnt, 1u) == pieces - 1 ? 1u : 0u;
      named_bar_sync(1, 128);
      if (*last_flag != 0u) {
        __threadfence();
        // the pieces in k order (piece p from pair c_first + p, in the slot of its
        // first piece when its run starts inside this tile); this CTA's own piece
        // comes from TMEM
        const uint32_t own = pair - c_first;
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
        if (row == 0) *cnt = 0u;  // ready for the next launch
      }
      release(acc);
    }
  }

  // Neither CTA frees its tensor memory, or exits, while the other may still touch
  // its shared memory, barriers or tensor memory.
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

// Pairs that can be resident at once (one CTA per SM), per device.
int resident_pairs(int num_sms) {
  static std::atomic<int> cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return num_sms / 2;
  if (dev < 64 && cached[dev].load(std::memory_order_relaxed) > 0) return cached[dev].load();
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (num_sms / 2), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kBytes + 1024;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, dw_gemm_kernel, &cfg) != cudaSuccess || n <= 0)
    n = num_sms / 2;
  if (n > num_sms / 2) n = num_sms / 2;
  if (dev < 64) cached[dev].store(n);
  return n;
}

}  // namespace

size_t dw_smem_bytes() { return kBytes + 1024; }

// Order of the device's dW launches (they share the workspace above): the event
// of the last launch, and whether there was one.
constexpr int kOrderDevices = 64;
static std::mutex g_dw_order_mu;
static cudaEvent_t g_dw_done[kOrderDevices] = {};
static bool g_dw_launched[kOrderDevices] = {};

cudaError_t reset_dw_counters() {
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_dw_cnt);
  if (e != cudaSuccess) return e;
  return cudaMemset(p, 0, sizeof(g_dw_cnt));
}

cudaError_t launch_dw_gemm(const CUtensorMap& tmap_x, const CUtensorMap& tmap_dy,
                           const DwArgs& a, int num_sms, cudaStream_t stream) {
  const size_t smem = dw_smem_bytes();
  cudaError_t e = ensure_smem_limit<dw_gemm_kernel>(static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int64_t tiles = ((a.k + kDwPairK - 1) / kDwPairK) * ((a.n + kDwTileN - 1) / kDwTileN);
  int64_t pairs = resident_pairs(num_sms);
  if (pairs > tiles) pairs = tiles;
  if (pairs > kDwMaxCtas / 2) pairs = kDwMaxCtas / 2;
  if (pairs < 1) pairs = 1;
  // The stream-K workspace and counters are shared by the device's dW launches:
  // every launch after the first waits for the previous one, whatever stream
  // either was issued on (a wait on the same stream's own last event costs
  // nothing on the device). A launch captured into a CUDA graph may not depend on
  // work outside the capture: there the graph's own edges order the dW nodes, and
  // the event is neither waited on nor recorded.
  std::lock_guard<std::mutex> lock(g_dw_order_mu);
  int dev = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if (dev >= kOrderDevices) return cudaErrorInvalidDevice;
  cudaStreamCaptureStatus capture = cudaStreamCaptureStatusNone;
  if ((e = cudaStreamIsCapturing(stream, &capture)) != cudaSuccess) return e;
  if (capture != cudaStreamCaptureStatusNone) {
    dw_gemm_kernel<<<static_cast<unsigned>(2 * pairs), kThreads, smem, stream>>>(tmap_x, tmap_dy, a);
    return cudaGetLastError();
  }
  if (g_dw_done[dev] == nullptr &&
      (e = cudaEventCreateWithFlags(&g_dw_done[dev], cudaEventDisableTiming)) != cudaSuccess)
    return e;
  if (g_dw_launched[dev] && (e = cudaStreamWaitEvent(stream, g_dw_done[dev], 0)) != cudaSuccess)
    return e;
  dw_gemm_kernel<<<static_cast<unsigned>(2 * pairs), kThreads, smem, stream>>>(tmap_x, tmap_dy, a);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if ((e = cudaEventRecord(g_dw_done[dev], stream)) != cudaSuccess) return e;
  g_dw_launched[dev] = true;
  return cudaSuccess;
}

}  // namespace tq
