// decode.cu — W1.58A16 forward for few tokens (m <= 16): an HBM-streaming kernel
// over the packed codes of one or many matrices in one launch (§8: at small batch
// the layer is bound by weight traffic; 2-bit codes + fp32 group scales are 0.28
// bytes per weight at g = 128).
//
// Work unit = a block of 256 consecutive weight rows of one matrix over its
// whole K. Per CTA (one per SM) a producer warp takes unit blockIdx.x first (no
// claim latency before the first load), then claims units one at a time from
// a per-launch global counter, in order, with the matrices of the batch sorted
// by decreasing K (the last units claimed are the shortest; SMs do not all
// receive HBM data at the same rate, so static shares leave SMs idle). It
// streams each unit as segments of 256 rows x 512 k: the 32 KB of codes are one
// 2-D TMA load of 128-byte rows with the 128-byte swizzle (which halves the
// consumers' bank conflicts; rows past n and columns past k read as zero;
// narrower rows cost the TMA unit as much per row and halved the stream rate),
// completing on the segment's "full" mbarrier. The group scales of a unit come
// apart from the segments, into two buffers that alternate: with at most 32
// groups per row the unit's rows are contiguous and arrive in one bulk copy;
// with more, a 2-D TMA box of the unit's 256 rows x 32 groups (128-byte rows,
// 128-byte swizzle, so that the eight rows a warp reads fall on distinct banks)
// covers the next 32·g of k — eight segments at g = 128 — where per-segment
// copies of each row's few scales had halved the stream. Only when the rows are
// not a multiple of 16 bytes (k/g % 4 != 0) do the producer's 32 lanes copy each
// segment's scales into its slot with 4-byte cp.async. TMA keeps a ring of stages
// segments (~100 KB per SM) in flight without holding registers or load-unit
// slots — per-lane cp.async streaming tops out near half of HBM bandwidth here.
//
// Consumer warps own 32 rows of the block (two m16 row tiles that share every
// activation fragment) over the whole K, so their accumulators persist across the
// unit's segments; up to 8 tokens two warps share each 32-row slice (each takes
// half of every segment's chunks, four consumer warps per scheduler) and add
// their partial sums once per unit through shared memory.
// Per 128-wide chunk of a segment (four per segment) a warp runs eight
// mma.sync.m16n8k16 (bf16 in, fp32 accumulate) per row tile with the expanded
// weights as the 16 x 16 A operand and up to 8 tokens as the n8 B operand (two B
// tiles for 9..16 tokens). The reduction index of the MMA is permuted identically on both
// operands so that lane (g, t) (g = lane / 4, t = lane % 4) consumes exactly code
// words t and t + 4 of the chunk (k offsets 16t .. 16t + 15 and 64 + 16t .. 64 + 16t
// + 15) for rows g and g + 8, and x[token g] at the same offsets: MMA kb takes word
// w = t (kb < 4) or t + 4 (kb >= 4), offsets 16w + 4 (kb % 4) + {0,1} for fragment
// slots (2t, 2t+1) and + {2,3} for slots (2t+8, 2t+9). Tokens past m read token
// m - 1: their output columns are never stored, and MMA columns do not mix.
//
// Pieces of k: a launch with fewer blocks of 256 rows than SMs (one layer's
// projection at a time) runs clusters of P = 8, 4 or 2 CTAs instead of the
// persistent grid, one cluster per block, CTA p streaming segments [p nseg / P,
// (p + 1) nseg / P); the other CTAs send their fp32 partial sums (the lanes that
// hold tokens below m) into the first CTA's shared memory with st.async, counted on
// its barrier, and the first CTA adds them to its own in piece order before the
// store — the same sums in the same order on every run.
//
// Every launch is a programmatic dependent launch: its CTAs may start on SMs the
// previous grid on the stream leaves free, set up, prefetch their first unit's
// codes and scales into L2 (coherent with any write still to come), and then wait
// for that grid before any other global access.
//
// Expansion: pair j of a code word -> bf16x2 (2c, 2c) by ((w << (14 - 2j)) &
// 0xC000C000) (layout of include/tq.h). For g >= 128 a chunk lies in one group:
// each group's products are accumulated from zero and folded into the output
// with the exact fp32 scale s, the sums halved (exactly) at the store. For g <= 64
// the groups of a chunk meet inside one MMA, so the expansion multiplies by
// bf16(s)/2 as the prefill kernels do.
//
// A consumer warp reads a unit's descriptor once, at its first segment, and takes
// every per-matrix decision there (scale addressing, exact or bf16 scaling, which
// segments need range guards); per segment it runs one wait, its chunks and one
// arrival.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <type_traits>

#include "decode.cuh"
#include "kernels.cuh"
#include "ptx.cuh"

namespace tq {
namespace {

constexpr int kRows = kDecodeRows;               // rows per unit (16 per consumer warp)
constexpr int kTiles = 2;                          // m16 row tiles per consumer warp
constexpr int kRowWarps = kRows / (16 * kTiles);   // warps covering the unit's rows
// Up to 8 tokens two warps share each 32-row slice, one per half of every
// segment's chunks (four consumer warps per scheduler); 9..16 tokens need the
// registers of one warp per slice.
template <bool kTwoTiles>
struct DecodeCfg {
  static constexpr int kSplit = kTwoTiles ? 1 : 2;
  static constexpr int kConsumers = kRowWarps * kSplit;
  static constexpr int kThreads = (kConsumers + 1) * 32;  // + one producer warp
};
constexpr int kRedBytes = 2 * kRowWarps * 32 * kTiles * 4 * 4;  // partial sums, two units
// Launches that cut k into P pieces: the first CTA of a cluster receives the
// partial sums of the other P - 1, [piece - 1][row warp][lane][8 floats, or 16
// with two n-tiles].
template <bool kTwoTiles>
__host__ __device__ constexpr int xpart_lane_floats() { return kTwoTiles ? 16 : 8; }
// Bytes one CTA sends for one row warp: 32 (two float4, one per row tile) from
// each of the 8 lanes of every t with tokens 2t, 2t + 1 below m, and as much for
// tokens 8 + 2t, 9 + 2t with two n-tiles.
template <bool kTwoTiles>
__host__ __device__ constexpr int xpart_slice_bytes(int m) {
  return 8 * 32 * (((m < 8 ? m : 8) + 1) / 2 +
                   (kTwoTiles && m > 8 ? (m - 8 + 1) / 2 : 0));
}
__host__ __device__ constexpr int xpart_bytes(bool two_tiles, int pieces) {
  return pieces > 1 ? (pieces - 1) * kRowWarps * 32 * (two_tiles ? 16 : 8) * 4 : 0;
}
// (the hand-off area exists only where two warps share a row slice)
template <bool kTwoTiles>
__host__ __device__ constexpr int red_bytes() { return kTwoTiles ? 0 : kRedBytes; }
constexpr int kSegK = kDecodeSegK;               // k per segment (one TMA box of 32 words)
constexpr int kChunks = kSegK / 128;             // 128-wide chunks per segment
constexpr int kCodeBytes = kRows * kSegK / 4;    // 32 KB
// x of one token over a segment (1 KB), tokens 1040 bytes apart (= 16 mod 128) so
// that the two tokens of a quarter-warp read disjoint shared-memory banks.
constexpr int kXTokBytes = kSegK * 2 + 16;
constexpr int kMaxStages = 8;
constexpr int kHeadBytes = 1024;                 // barriers and segment descriptors
constexpr int kSmemLimit = 227 * 1024;
// Slot layout (sizes set per launch from the batch's group sizes and m):
// [codes 32 KB][scales: 256 rows x the segment's groups (4-byte mode only)]
// [x: m tokens x kSegK]

static_assert(kRowWarps == 8, "two m16 row tiles per row warp");
static_assert(kCodeBytes == 32 * 1024, "codes box");
static_assert(sizeof(DecodeBatch) <= 32764, "kernel parameter space");
static_assert(kDecodeWinGroups * 4 == 128, "a window row is one 128-byte swizzle row");

// Row strides (in floats) of the scale areas. The eight rows a warp reads at once
// (rows = 0..7 mod 8) fall on distinct banks when the stride is odd, as in the
// 4-byte mode, whose producer copies rows one by one. A unit's scales arrive in
// one bulk copy and keep their rows gpr apart (per-row copies into padded rows
// cost more than the bank conflicts they remove). A window's rows are 32 floats
// apart with 16-byte chunk j of row r at chunk j ^ (r % 8) (the TMA 128-byte
// swizzle): float q of row r sits at 32 r + (q ^ 4 (r % 8)).
__host__ __device__ constexpr int unit_scale_stride(int gpr) { return gpr; }
__host__ __device__ constexpr int seg_scale_stride(int log2g) {
  return (log2g >= 9 ? 1 : kSegK >> log2g) | 1;
}

// Segment descriptor written by the producer next to the slot's barriers; it
// carries what the consumers need of the matrix, so they never index the
// parameter table.
struct SegInfo {
  int32_t mat;    // matrix of the batch; -1: end of the stream
  int32_t row0;   // first row of the unit
  int32_t seg;    // segment index along k
  int32_t s1;     // end of the unit's segments (exclusive; its first is seg of its first stage)
  int32_t k;      // reduction length
  int32_t n;      // rows of the matrix
  int32_t log2g;
  int32_t mode;   // scale fetch mode | y_bf16 << 8
  void* y;        // output [m][n]
  int64_t pad;
};
static_assert(sizeof(SegInfo) == 48, "segment descriptor");

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

// Pair j of a code word as a bf16x2 of (2c, 2c): the mask keeps the pair's two
// fields, the multiplication by mul = 2^(14 - 2j) moves them to bits 14-15 and
// 30-31 (exact, the fields are 16 bits apart). mul is a register whose value the
// compiler does not see, so the move runs as an integer multiply on the FMA pipe
// instead of a shift on the ALU pipe, which the mask already loads.
// Pair 7 already sits at bits 14-15 and 30-31: the mask alone.
__device__ __forceinline__ uint32_t pair_bits(uint32_t w, int j, uint32_t mul) {
  if (j == 7) return w & 0xC000C000u;
  return (w & (0x00030003u << (2 * j))) * mul;
}

__device__ __forceinline__ uint32_t opaque(uint32_t v) {
  uint32_t r;
  asm volatile("mov.b32 %0, %1;" : "=r"(r) : "r"(v));
  return r;
}

// mma.sync m16n8k16, A and B in the activation type (both bf16, or both fp16). Not
// volatile: the compiler may interleave the independent chains of a warp.
template <bool F16>
__device__ __forceinline__ void mma16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  if constexpr (F16)
    asm(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  else
    asm(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// The same with a zero accumulator input.
template <bool F16>
__device__ __forceinline__ void mma16816_zc(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                            uint32_t a3, uint32_t b0, uint32_t b1) {
  if constexpr (F16)
    asm(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%10, %10, %10, %10};"
        : "=f"(c[0]), "=f"(c[1]), "=f"(c[2]), "=f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(0.0f));
  else
    asm(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%10, %10, %10, %10};"
        : "=f"(c[0]), "=f"(c[1]), "=f"(c[2]), "=f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(0.0f));
}

// 4-byte global -> shared copy; zero-filled when src_bytes is 0.
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}

// Arrive on `bar` once every cp.async this thread issued so far has landed; the
// arrival counts toward the barrier's expected count.
__device__ __forceinline__ void cp_async_arrive(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

// s / 2 rounded to the activation type, in both halves.
template <bool F16>
__device__ __forceinline__ uint32_t half_scale_x2(float s) {
  uint32_t u;
  if constexpr (F16)
    u = __half_as_ushort(__float2half_rn(0.5f * s));
  else
    u = __bfloat16_as_ushort(__float2bfloat16_rn(0.5f * s));
  return u | (u << 16);
}

// Wait, with cluster-scope acquire, for a phase completed from other CTAs of the
// cluster (the bytes of their st.async stores into this CTA's shared memory), so
// that this thread's later reads see those bytes. Gives up like mbar_wait.
__device__ __forceinline__ bool mbar_test_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool lanes_wait_cluster(uint32_t bar, uint32_t parity, int* status) {
  bool ok = mbar_test_wait_cluster(bar, parity);
  if (!ok) {
    const uint64_t t0 = globaltimer_ns();
    const uint64_t limit = wait_limit_ns(status);
    for (uint32_t n = 1;; ++n) {
      if (mbar_test_wait_cluster(bar, parity)) {
        ok = true;
        break;
      }
      if ((n & 255u) == 0 && (globaltimer_ns() - t0 > limit || n >= kWaitMaxPolls)) {
        atomicExch(status, kStatusTimeout);
        break;
      }
    }
  }
  return __all_sync(0xffffffffu, ok);
}

// The cluster barrier in two halves: every thread arrives once the barriers are
// set up; a warp about to touch another CTA's shared memory waits for all
// arrivals, which also means that every CTA has started.
__device__ __forceinline__ void cluster_arrive() {
  // relaxed: the barrier set-up it covers was released by fence.mbarrier_init
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// 16 bytes into another CTA's shared memory, counted on that CTA's mbarrier
// (addresses from map_to_rank): the barrier's phase completes once all the bytes
// it expects have landed.
__device__ __forceinline__ void st_async_f4(uint32_t cluster_addr, float4 v, uint32_t cluster_bar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
          cluster_addr),
      "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(cluster_bar)
      : "memory");
}

// Programmatic dependent launch. launch_dependents lets the next launch on the stream
// (one made with the programmatic-serialisation attribute) start its CTAs on SMs
// that this grid leaves free; wait holds this thread until the previous grid on
// the stream has completed and its writes are visible.
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// L2 prefetches (no shared memory written, no barrier): L2 is where the device's
// writes meet, so a line fetched before the previous grid has finished writing it
// is updated in place and later loads see the new data.
__device__ __forceinline__ void prefetch_l2_tile(const CUtensorMap* map, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
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

// Unit scheduler of one launch: {next unit, CTAs done}. Zero at the start of a
// launch; the last CTA to finish claiming puts both back to zero. Launches take
// the slots in turn, so up to kSchedSlots launches may be in flight at once.
constexpr int kSchedSlots = 256;
__device__ uint32_t g_dsched[kSchedSlots][2];

// Test flag (tq_test_hooks, DeviceCtl word 1): in a launch cut into pieces of k, CTA 1
// sends none of its partial sums, so its cluster's first CTA waits for them in vain.
constexpr int kWithholdDecodePieces = 4;

// kPieces: a launch that cuts k into pieces (clusters; b.pieces > 1); without it
// the persistent grid, compiled with none of the pieces' code.
template <bool kTwoTiles, bool F16, bool kPieces>
__global__ void __launch_bounds__(DecodeCfg<kTwoTiles>::kThreads, 1)
    decode_kernel(const __grid_constant__ DecodeBatch b, uint32_t* sched) {
  constexpr int kConsumers = DecodeCfg<kTwoTiles>::kConsumers;
  constexpr int kSplit = DecodeCfg<kTwoTiles>::kSplit;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* head = align_shared<1024>(smem_raw);
  const int ub_bytes = b.ubuf_bytes;       // one unit-scale buffer (0: none in this launch)
  float* red = reinterpret_cast<float*>(head + kHeadBytes);  // [2][kRowWarps][32][8]
  const int pieces = kPieces ? b.pieces : 1;  // pieces of k per block of rows (cluster size)
  float* xpart = reinterpret_cast<float*>(head + kHeadBytes + red_bytes<kTwoTiles>());
  uint8_t* ubuf = reinterpret_cast<uint8_t*>(xpart) + xpart_bytes(kTwoTiles, pieces);
  uint8_t* smem = ubuf + 2 * ub_bytes;     // the ring
  const int stages = b.stages;
  const int slot_bytes = b.slot_bytes;
  const int scale_bytes = b.scale_bytes;
  const uint32_t ring = smem_u32(smem);
  const uint32_t bars = smem_u32(head);
  auto full_bar = [&](int s) { return bars + 8 * s; };
  auto empty_bar = [&](int s) { return bars + 8 * (kMaxStages + s); };
  auto sfull_bar = [&](int i) { return bars + 8 * (2 * kMaxStages + i); };
  auto sempty_bar = [&](int i) { return bars + 8 * (2 * kMaxStages + 2 + i); };
  // partial-sum hand-off between the two warps of a row slice, per buffer
  auto rfull_bar = [&](int w, int p) { return bars + 160 + 8 * (2 * w + p); };
  auto rempty_bar = [&](int w, int p) { return bars + 288 + 8 * (2 * w + p); };
  // pieces of k: in the first CTA of a cluster, "the other CTAs' partial sums of
  // row warp w have landed"; in the others, "the first CTA has them all" (this CTA
  // may leave)
  auto xfull_bar = [&](int w) { return bars + 416 + 8 * w; };
  auto xdone_bar = [&](int w) { return bars + 896 + 8 * w; };
  SegInfo* info = reinterpret_cast<SegInfo*>(head + 512);  // kMaxStages x 48 bytes
  int* status = b.status;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int m = b.m;

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(full_bar(s), 1 + 32);  // TMA expect_tx + an arrival per producer lane
      mbar_init(empty_bar(s), kConsumers);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(sfull_bar(i), 1);
      mbar_init(sempty_bar(i), kConsumers);
    }
    for (int w = 0; w < kRowWarps; ++w)
      for (int p = 0; p < 2; ++p) {
        mbar_init(rfull_bar(w, p), 1);
        mbar_init(rempty_bar(w, p), 1);
      }
    if (pieces > 1)
      for (int w = 0; w < kRowWarps; ++w) {
        // completed by the bytes the other CTAs store (the one arrival is this one)
        mbar_init(xfull_bar(w), 1);
        mbar_arrive_expect_tx(xfull_bar(w), (pieces - 1) * xpart_slice_bytes<kTwoTiles>(m));
        mbar_init(xdone_bar(w), 1);
      }
    fence_mbar_init();
  }
  __syncthreads();
  // Every CTA of the cluster has started and set up its barriers once the cluster
  // barrier completes: arrive now, wait only before the first access to another
  // CTA's shared memory (long since complete by then).
  if (pieces > 1) cluster_arrive();
  // the next decode launch on the stream may start its CTAs on the SMs this grid
  // leaves free; they prefetch into L2 and then wait for this grid (pdl_wait)
  pdl_launch_dependents();

  if (warp == kConsumers) {
    // ------------------------------------------------------------ producer
    const uint64_t stream_policy = policy_evict_first();  // codes and scales: read once
    const uint64_t keep_policy = policy_evict_last();     // x: read by every unit
    int slot = 0;
    uint32_t parity = 0;
    int64_t issued = 0;
    int units_u = 0;  // units and windows whose scales went through the buffers
    bool ok = true;
    int claims = 0;
    if (lane == 0 && static_cast<int>(blockIdx.x) < b.total_units) {
      // Before the previous grid on the stream has finished: bring this CTA's first
      // unit's codes (as many segments as the ring holds) and scales into L2.
      const int u = static_cast<int>(blockIdx.x);
      const int d = find_mat(b, u);
      const DecodeMat& mt = b.mats[d];
      const int nseg = static_cast<int>((mt.k + kSegK - 1) / kSegK);
      const int local = u - mt.unit0;
      const int piece = local % pieces;
      const int64_t row0 = static_cast<int64_t>(local / pieces) * kRows;
      const int s0 = piece * nseg / pieces, s1 = (piece + 1) * nseg / pieces;
      for (int s = s0; s < s1 && s < s0 + stages; ++s)
        prefetch_l2_tile(&b.maps[d], s * (kSegK / 16), static_cast<int32_t>(row0));
      const int64_t gpr = mt.k >> mt.log2g;
      if (mt.scale_mode == kDecodeScaleUnit) {
        const int64_t rows = mt.n - row0 < kRows ? mt.n - row0 : kRows;
        prefetch_l2(mt.scales + row0 * gpr, static_cast<uint32_t>(rows * gpr * 4));
      } else if (mt.scale_mode == kDecodeScaleWin) {
        prefetch_l2_tile(&b.maps[mt.smap], (s0 >> (mt.log2g - 4)) * kDecodeWinGroups,
                         static_cast<int32_t>(row0));
      }
    }
    pdl_wait();  // nothing of the previous grid's output is read or overwritten before
    for (;;) {
      // the first unit of every CTA is dealt (blocks <= units), later ones claimed
      // (with pieces of k every CTA takes its one dealt unit)
      int u = static_cast<int>(blockIdx.x);
      if (claims++ > 0) {
        if (pieces > 1) break;
        if (lane == 0) u = static_cast<int>(gridDim.x + atomicAdd(&sched[0], 1u));
        u = __shfl_sync(0xffffffffu, u, 0);
      }
      if (u >= b.total_units) break;
      const int d = find_mat(b, u);
      const DecodeMat& mt = b.mats[d];
      const int nseg = static_cast<int>((mt.k + kSegK - 1) / kSegK);
      // unit = (block of rows, piece of k): piece p of P takes segments
      // [p nseg / P, (p + 1) nseg / P), none empty (the launcher keeps P <= nseg)
      const int local = u - mt.unit0;
      const int piece = local % pieces;
      const int64_t row0 = static_cast<int64_t>(local / pieces) * kRows;
      const int s0 = piece * nseg / pieces, s1 = (piece + 1) * nseg / pieces;
      const int log2g = mt.log2g;
      const int64_t gpr = mt.k >> log2g;               // groups per row
      const int ng = log2g >= 9 ? 1 : kSegK >> log2g;  // scales per row per segment
      // scales through the two unit buffers: the whole unit at once, or a window of
      // kDecodeWinGroups groups (2^(log2g - 4) segments) at a time
      const bool win = mt.scale_mode == kDecodeScaleWin;
      // segment s opens a buffer at the unit's first segment and, in the window
      // mode, when s & wmask == 0 (windows of 32 groups from group 0, every
      // 2^(log2g - 4) segments)
      const int wmask = win ? (1 << (log2g - 4)) - 1 : 0x7fffffff;
      auto scales_to_buffer = [&](int s) -> bool {
        const int ub = units_u & 1;
        if (units_u >= 2 && !warp_wait(sempty_bar(ub), ((units_u >> 1) + 1) & 1, status))
          return false;
        if (lane == 0) {
          const uint32_t dst = smem_u32(ubuf + ub * ub_bytes);
          if (win) {
            // rows past n and groups past k/g read as zero
            mbar_arrive_expect_tx(sfull_bar(ub), kRows * kDecodeWinGroups * 4);
            tma_load_2d_hint(dst, &b.maps[mt.smap], sfull_bar(ub),
                             (s >> (log2g - 4)) * kDecodeWinGroups, static_cast<int32_t>(row0),
                             stream_policy);
          } else {
            // rows past n are not copied; their outputs are never stored
            const int64_t rows = mt.n - row0 < kRows ? mt.n - row0 : kRows;
            const uint32_t bytes = static_cast<uint32_t>(rows * gpr * 4);
            mbar_arrive_expect_tx(sfull_bar(ub), bytes);
            bulk_load(dst, mt.scales + row0 * gpr, bytes, sfull_bar(ub), stream_policy);
          }
        }
        ++units_u;
        return true;
      };
      const bool buffered = win || mt.scale_mode == kDecodeScaleUnit;
      for (int s = s0; s < s1; ++s) {
        if (buffered && (s == s0 || (s & wmask) == 0) && !scales_to_buffer(s)) {
          ok = false;
          break;
        }
        if (issued >= stages && !warp_wait(empty_bar(slot), parity ^ 1u, status)) {
          ok = false;
          break;
        }
        const int64_t g0 = (static_cast<int64_t>(s) * kSegK) >> log2g;  // first group
        const uint32_t cdst = ring + slot * slot_bytes;
        const uint32_t sdst = cdst + kCodeBytes;
        const uint32_t xdst = sdst + scale_bytes;
        // the tokens' x over the segment's k (a multiple of 64, so of 128 bytes)
        const int64_t kx = mt.k - static_cast<int64_t>(s) * kSegK < kSegK
                               ? mt.k - static_cast<int64_t>(s) * kSegK : kSegK;
        const uint32_t xbytes = static_cast<uint32_t>(kx) * 2u;
        if (lane == 0) {
          info[slot] = SegInfo{d, static_cast<int32_t>(row0), s, s1,
                               static_cast<int32_t>(mt.k), static_cast<int32_t>(mt.n),
                               log2g, mt.scale_mode | (mt.y_bf16 << 8), mt.y, 0};
          mbar_arrive_expect_tx(full_bar(slot), kCodeBytes + static_cast<uint32_t>(m) * xbytes);
          tma_load_2d_hint(cdst, &b.maps[d], full_bar(slot), s * (kSegK / 16),
                           static_cast<int32_t>(row0), stream_policy);
        }
        __syncwarp();
        if (lane < m)
          bulk_load(xdst + lane * kXTokBytes,
                    static_cast<const uint16_t*>(mt.x) + lane * mt.k +
                        static_cast<int64_t>(s) * kSegK,
                    xbytes, full_bar(slot), keep_policy);
        if (buffered) {
          mbar_arrive(full_bar(slot));
        } else {
          // [256 rows][ng] from group g0 (rows seg_scale_stride apart), zero past n
          // and past k
          const int ss = seg_scale_stride(log2g);
          for (int i = 0; i < kRows / 32; ++i) {
            const int r = lane + 32 * i;
            const int64_t row = row0 + r;
            for (int q = 0; q < ng; ++q) {
              const bool in = row < mt.n && g0 + q < gpr;
              const float* src = mt.scales + (in ? row * gpr + g0 + q : 0);
              cp_async4(sdst + (r * ss + q) * 4, src, in ? 4u : 0u);
            }
          }
          cp_async_arrive(full_bar(slot));
        }
        ++issued;
        if (++slot == stages) {
          slot = 0;
          parity ^= 1u;
        }
      }
      if (!ok) break;
    }
    if (ok) {
      // end of the stream: a stage with no data tells the consumers
      if (issued >= stages && !warp_wait(empty_bar(slot), parity ^ 1u, status)) ok = false;
      if (ok) {
        if (lane == 0) info[slot].mat = -1;
        __syncwarp();
        mbar_arrive(full_bar(slot));  // 32 lanes
        if (lane == 0) mbar_arrive(full_bar(slot));
      }
    }
    // this CTA claims no more: the last CTA to get here resets the scheduler
    if (lane == 0) {
      __threadfence();
      if (atomicAdd(&sched[1], 1u) == gridDim.x - 1) {
        atomicExch(&sched[0], 0u);
        atomicExch(&sched[1], 0u);
      }
    }
    // Nothing may still write this CTA's shared memory when it exits: normally
    // the consumers waited for every copy; if a wait gave up, wait here for the
    // segments issued last (no end marker was written on this path) and for the
    // unit-scale copies.
    if (!ok && lane == 0) {
      for (int64_t j = issued > stages ? issued - stages : 0; j < issued; ++j)
        if (!mbar_wait(full_bar(static_cast<int>(j % stages)),
                       static_cast<uint32_t>((j / stages) & 1), status))
          break;
      for (int j = units_u > 2 ? units_u - 2 : 0; j < units_u; ++j)
        if (!mbar_wait(sfull_bar(j & 1), (j >> 1) & 1, status)) break;
    }
    if (!ok) asm volatile("cp.async.wait_all;" ::: "memory");
    return;
  }

  // -------------------------------------------------------------- consumers
  pdl_wait();  // (their outputs may be read by the previous grid until it completes)
  // Warp w owns rows 32wr .. 32wr + 31 of the unit (wr = w % 8) as two m16 tiles
  // that share every activation fragment, over the chunks c of each segment with
  // c / (4 / kSplit) == w / 8; lane (g, t) holds rows 32wr + 16r + g (+8) of tile r.
  const int wr = warp % kRowWarps;
  const int kh = warp / kRowWarps;  // which part of every segment's chunks
  const int g = lane >> 2, t = lane & 3;
  uint32_t mul[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) mul[j] = opaque(1u << (14 - 2 * j));
  float acc[kTiles][4], acc1[kTiles][4];  // tokens 0..7 and 8..15
#pragma unroll
  for (int r = 0; r < kTiles; ++r)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[r][i] = acc1[r][i] = 0.f;
  const int tok0 = g < m ? g : m - 1;  // tokens past m read token m - 1
  const int tok1 = g + 8 < m ? g + 8 : m - 1;
  const int rl = 32 * wr + g;          // row of tile 0 for C slots 0, 1 (+8: slots 2, 3)
  // Lane t takes code words t and t + 4 of a chunk's eight (k offsets 16t ..
  // 16t + 15 and 64 + 16t .. 64 + 16t + 15): the 128-byte swizzle moves 16-byte
  // chunk j of row r to j ^ (r % 8), so one 32-bit load per word reaches all 32
  // banks across the warp's eight rows, and the x fragments of the four lanes of
  // a quarter-warp (bytes 32t .. 32t + 31 of each half chunk) fall on disjoint
  // banks too.
  constexpr int kMine = kChunks / kSplit;  // chunks of a segment this warp takes
  auto code_at = [&](int c) { return rl * (kSegK / 4) + (((2 * c) ^ g) << 4) + 4 * t; };  // word t
  const int dw4 = (g & 1) ? -16 : 16;  // word t + 4: 16-byte chunk (2c + 1) ^ g = ((2c) ^ g) ^ 1
  auto x_at = [&](int tok, int c) { return tok * kXTokBytes + 256 * c + 32 * t; };
  // kept in registers up to 8 tokens; recomputed per chunk with two n-tiles,
  // whose accumulators need the registers
  int code_off[kMine], x0_off[kMine];
#pragma unroll
  for (int cc = 0; cc < kMine; ++cc) {
    code_off[cc] = code_at(kh * kMine + cc);
    x0_off[cc] = x_at(tok0, kh * kMine + cc);
  }
  int units_r = 0;  // units whose partial sums were handed over
  int units_u = 0;  // units and windows whose scales came through the buffers
  int slot = 0;
  uint32_t parity = 0;
  for (;;) {
    // The first segment of a unit carries the unit's descriptor: everything that
    // depends on the matrix is decided here once, so that per segment a warp runs
    // one wait, its chunks and one arrival.
    if (!lanes_wait(full_bar(slot), parity, status)) return;
    const SegInfo si = info[slot];
    if (si.mat < 0) break;
    const int k = si.k;
    const int log2g = si.log2g;
    const int mode = si.mode & 0xff;
    const bool unit_scales = mode == kDecodeScaleUnit;
    const bool win_scales = mode == kDecodeScaleWin;
    const int nfull = k / kSegK;  // segments that lie inside k
    // this unit's piece of the segments (all of them without pieces)
    const int s0 = kPieces ? si.seg : 0;
    const int s1 = kPieces ? si.s1 : (k + kSegK - 1) / kSegK;
    // a window spans 2^(log2g - 4) segments (32 groups of g): segment s opens one
    // when s & wmask == 0 and closes it when s & wmask == wmask (or s is the last)
    const int wmask = (1 << (log2g - 4)) - 1;
    // Scale of unit row r and group q: area[r * sstride + sq(q) - sq0], the area
    // being the unit buffer (sq(q) = q, sq0 = 0), the segment's slot (sq(q) = q, sq0 =
    // its first stored group) or the window buffer (sq(q) = (q & 31) ^ qx, sq0 = 0:
    // the swizzle of row r is 4 (r % 8), and this lane's rows are all g mod 8).
    const int sstride = unit_scales ? unit_scale_stride(k >> log2g)
                        : win_scales ? kDecodeWinGroups
                                     : seg_scale_stride(log2g);
    const int qx = g << 2;
    const float* ubase = nullptr;
    if (unit_scales) {
      const int ub = units_u & 1;
      if (!lanes_wait(sfull_bar(ub), (units_u >> 1) & 1, status)) return;
      ubase = reinterpret_cast<const float*>(ubuf + ub * ub_bytes);
    }
    // scale offsets of this lane's rows: tile r, C slots 0-1 (h = 0) and 2-3 (h = 1)
    int soff[kTiles][2];
#pragma unroll
    for (int r = 0; r < kTiles; ++r)
#pragma unroll
      for (int h = 0; h < 2; ++h) soff[r][h] = (rl + 16 * r + 8 * h) * sstride;
#pragma unroll
    for (int r = 0; r < kTiles; ++r)
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[r][i] = acc1[r][i] = 0.f;

    // Segment s of the unit: its wait (the first one's was the descriptor's), this
    // warp's chunks, the release of the slot. kGuard: the segment reaches past k.
    // kKind 1 (g = 128) and 2 (g >= 256): a chunk lies in one group; its products
    // are accumulated from zero and folded in with the fp32 scale s (the expanded
    // codes are 2c, so the sums are twice the output, halved exactly at the store).
    // kKind 0 (g = 32, 64): the lane's words t and t + 4 each lie in one group,
    // whose bf16(s)/2 multiplies the expanded pairs.
    auto segment = [&](int s, auto guard, auto kind, auto win) -> bool {
      constexpr bool kGuard = decltype(guard)::value;
      constexpr int kKind = decltype(kind)::value;
      constexpr bool kWin = decltype(win)::value;  // the matrix takes scale windows
      auto sq = [&](int q) { return kWin ? (q & (kDecodeWinGroups - 1)) ^ qx : q; };
      if (s > s0 && !lanes_wait(full_bar(slot), parity, status)) return false;
      if (kWin && (s == s0 || (s & wmask) == 0)) {
        const int ub = units_u & 1;
        if (!lanes_wait(sfull_bar(ub), (units_u >> 1) & 1, status)) return false;
        ubase = reinterpret_cast<const float*>(ubuf + ub * ub_bytes);
      }
      const uint8_t* cbase = smem + slot * slot_bytes;
      const int kseg = s * kSegK + 128 * kMine * kh;  // first k of this warp's chunks
      const int g0 = (s * kSegK) >> log2g;             // first group of the segment
      const float* sl = unit_scales || kWin
                            ? ubase
                            : reinterpret_cast<const float*>(cbase + kCodeBytes) - g0;
      // scales of group q0 + dq(cc) for the lane's four rows: sp[r][h][sq(q0 + dq)]
      const float* sp[kTiles][2];
      const int q0 = kseg >> log2g;
#pragma unroll
      for (int r = 0; r < kTiles; ++r)
#pragma unroll
        for (int h = 0; h < 2; ++h) sp[r][h] = sl + soff[r][h];
      // g = 128, two chunks per warp: the scales of their groups q0, q0 + 1 for all
      // four rows, loaded once. In the unit and window modes (row strides k/g and 32,
      // area bases on 4-group boundaries; q0 = 4s + 2kh is even, and the swizzle keeps
      // q0 and q0 + 1 side by side) one 8-byte load per row takes both: half the loads
      // (and, in the unit mode, half the bank conflicts: a load's eight rows sit 16 or
      // 32 words apart there; the window's swizzle has none). The 4-byte mode's odd
      // row stride (5) allows no 8-byte load and has no conflicts: two 4-byte loads.
      // Past k (last segment) the second value is not used.
      constexpr bool kPairScales = kKind == 1 && kMine == 2;
      float2 sv[kTiles][2];
      if constexpr (kPairScales) {
        const bool wide = mode != kDecodeScale4;
#pragma unroll
        for (int r = 0; r < kTiles; ++r)
#pragma unroll
          for (int h = 0; h < 2; ++h)
            sv[r][h] = wide ? *reinterpret_cast<const float2*>(sp[r][h] + sq(q0))
                            : make_float2(sp[r][h][q0], sp[r][h][q0 + 1]);
      }
      const uint8_t* xs = cbase + kCodeBytes + scale_bytes;  // x of the m tokens
#pragma unroll
      for (int cc = 0; cc < kMine; ++cc) {
        const int c = kh * kMine + cc;
        const int kc = kseg + 128 * cc;  // chunk start
        if (kGuard && kc >= k) break;
        // k is a multiple of 64: a chunk reaching past k has its first half inside
        const bool khi = !kGuard || kc + 128 <= k;  // the second half lies inside k
        // words t (.x) and t + 4 (.y) of rows rl + 16r (h = 0) and + 8 (h = 1)
        uint2 w[kTiles][2];
        const uint8_t* cw0 = cbase + (kTwoTiles ? code_at(c) : code_off[cc]);
        const uint8_t* cw1 = cw0 + dw4;
#pragma unroll
        for (int r = 0; r < kTiles; ++r)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            w[r][h].x = *reinterpret_cast<const uint32_t*>(cw0 + (16 * r + 8 * h) * (kSegK / 4));
            w[r][h].y = *reinterpret_cast<const uint32_t*>(cw1 + (16 * r + 8 * h) * (kSegK / 4));
          }
        // x of the lane's offsets, xv[0..1] for word t, xv[2..3] for word t + 4
        // (past k the slot holds no x)
        uint4 xv[4], yv[4];
        const uint8_t* xa = xs + (kTwoTiles ? x_at(tok0, c) : x0_off[cc]);
        const uint8_t* xb = xs + x_at(tok1, c);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int off = 16 * (i & 1) + 128 * (i >> 1);
          const bool in = i < 2 || khi;
          xv[i] = in ? *reinterpret_cast<const uint4*>(xa + off) : make_uint4(0, 0, 0, 0);
          if (kTwoTiles) yv[i] = in ? *reinterpret_cast<const uint4*>(xb + off) : make_uint4(0, 0, 0, 0);
        }
        const uint32_t* xr = reinterpret_cast<const uint32_t*>(xv);
        const uint32_t* yr = reinterpret_cast<const uint32_t*>(yv);
        if constexpr (kKind != 0) {
          float p[kTiles][4], p1[kTiles][4];
#pragma unroll
          for (int kb = 0; kb < 8; ++kb) {
            const int j = 2 * (kb & 3);
#pragma unroll
            for (int r = 0; r < kTiles; ++r) {
              const uint32_t u0 = kb < 4 ? w[r][0].x : w[r][0].y;
              const uint32_t u1 = kb < 4 ? w[r][1].x : w[r][1].y;
              const uint32_t a0 = pair_bits(u0, j, mul[j]), a1 = pair_bits(u1, j, mul[j]);
              const uint32_t a2 = pair_bits(u0, j + 1, mul[j + 1]);
              const uint32_t a3 = pair_bits(u1, j + 1, mul[j + 1]);
              if (kb == 0) {
                mma16816_zc<F16>(p[r], a0, a1, a2, a3, xr[0], xr[1]);
                if (kTwoTiles) mma16816_zc<F16>(p1[r], a0, a1, a2, a3, yr[0], yr[1]);
              } else {
                mma16816<F16>(p[r], a0, a1, a2, a3, xr[2 * kb], xr[2 * kb + 1]);
                if (kTwoTiles) mma16816<F16>(p1[r], a0, a1, a2, a3, yr[2 * kb], yr[2 * kb + 1]);
              }
            }
          }
          // group of chunk cc: q0 + cc for g = 128; for g >= 256 the chunks of a
          // warp's pair share a group (k offsets 256 kh + 128 cc of a 512-aligned
          // segment), with four chunks one group per two (g = 256) or one in all
          const int dq = kKind == 1 ? cc : (kMine <= 2 ? 0 : (128 * cc) >> log2g);
          // C slots 0, 1: row rl + 16r, slots 2, 3: row rl + 16r + 8
#pragma unroll
          for (int r = 0; r < kTiles; ++r) {
            const float h0 = kPairScales ? (cc == 0 ? sv[r][0].x : sv[r][0].y) : sp[r][0][sq(q0 + dq)];
            const float h1 = kPairScales ? (cc == 0 ? sv[r][1].x : sv[r][1].y) : sp[r][1][sq(q0 + dq)];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              acc[r][i] = fmaf(i < 2 ? h0 : h1, p[r][i], acc[r][i]);
              if (kTwoTiles) acc1[r][i] = fmaf(i < 2 ? h0 : h1, p1[r][i], acc1[r][i]);
            }
          }
        } else {
          // the lane's words t and t + 4 lie in groups qa and qb
          const int qa = (kc + 16 * t) >> log2g, qb = (kc + 64 + 16 * t) >> log2g;
#pragma unroll
          for (int r = 0; r < kTiles; ++r) {
            const uint32_t hs0a = half_scale_x2<F16>(sl[soff[r][0] + sq(qa)]);
            const uint32_t hs1a = half_scale_x2<F16>(sl[soff[r][1] + sq(qa)]);
            const uint32_t hs0b = khi ? half_scale_x2<F16>(sl[soff[r][0] + sq(qb)]) : 0u;
            const uint32_t hs1b = khi ? half_scale_x2<F16>(sl[soff[r][1] + sq(qb)]) : 0u;
#pragma unroll
            for (int kb = 0; kb < 8; ++kb) {
              const int j = 2 * (kb & 3);
              const uint32_t u0 = kb < 4 ? w[r][0].x : w[r][0].y;
              const uint32_t u1 = kb < 4 ? w[r][1].x : w[r][1].y;
              const uint32_t hs0 = kb < 4 ? hs0a : hs0b, hs1 = kb < 4 ? hs1a : hs1b;
              const uint32_t a0 = bmul2<F16>(pair_bits(u0, j, mul[j]), hs0);
              const uint32_t a1 = bmul2<F16>(pair_bits(u1, j, mul[j]), hs1);
              const uint32_t a2 = bmul2<F16>(pair_bits(u0, j + 1, mul[j + 1]), hs0);
              const uint32_t a3 = bmul2<F16>(pair_bits(u1, j + 1, mul[j + 1]), hs1);
              mma16816<F16>(acc[r], a0, a1, a2, a3, xr[2 * kb], xr[2 * kb + 1]);
              if (kTwoTiles) mma16816<F16>(acc1[r], a0, a1, a2, a3, yr[2 * kb], yr[2 * kb + 1]);
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty_bar(slot));
      if (kWin && ((s & wmask) == wmask || s + 1 == s1)) {
        if (lane == 0) mbar_arrive(sempty_bar(units_u & 1));  // after the __syncwarp
        ++units_u;
      }
      if (++slot == stages) {
        slot = 0;
        parity ^= 1u;
      }
      return true;
    };
    bool ok = true;
    auto run = [&](auto kind, auto win) {
      if constexpr (kTwoTiles) {
        // (two n-tiles: no register room for a second chunk body)
        for (int s = s0; s < s1 && ok; ++s) ok = segment(s, std::true_type{}, kind, win);
      } else {
        // the segments inside k, then the one reaching past k if this piece has it
        const int e = s1 < nfull ? s1 : nfull;
        for (int s = s0; s < e && ok; ++s) ok = segment(s, std::false_type{}, kind, win);
        if (ok && s1 > nfull) ok = segment(nfull, std::true_type{}, kind, win);
      }
    };
    auto run_kind = [&](auto kind) {
      if (win_scales)
        run(kind, std::true_type{});
      else
        run(kind, std::false_type{});
    };
    const bool exact = log2g >= 7;
    if (log2g == 7)
      run_kind(std::integral_constant<int, 1>{});
    else if (exact)
      run_kind(std::integral_constant<int, 2>{});
    else
      run_kind(std::integral_constant<int, 0>{});
    if (!ok) return;
    if (unit_scales) {
      if (lane == 0) mbar_arrive(sempty_bar(units_u & 1));
      ++units_u;
    }
    if (kSplit == 2) {
      // the second warp of the slice hands its partial sums to the first through
      // buffer units_r % 2 (bounded waits both ways: "written" and "read")
      const int pb = units_r & 1;
      const uint32_t ph = (units_r >> 1) & 1;
      float* rb = red + ((pb * kRowWarps + wr) * 32 + lane) * (kTiles * 4);
      if (kh == 1) {
        if (units_r >= 2 && !lanes_wait(rempty_bar(wr, pb), ph ^ 1u, status)) return;
#pragma unroll
        for (int r = 0; r < kTiles; ++r)
#pragma unroll
          for (int i = 0; i < 4; ++i) rb[r * 4 + i] = acc[r][i];
        __syncwarp();
        if (lane == 0) mbar_arrive(rfull_bar(wr, pb));
      } else {
        if (!lanes_wait(rfull_bar(wr, pb), ph, status)) return;
#pragma unroll
        for (int r = 0; r < kTiles; ++r)
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[r][i] += rb[r * 4 + i];
        __syncwarp();
        if (lane == 0) mbar_arrive(rempty_bar(wr, pb));
      }
      ++units_r;
    }
    if (kh == 0 && pieces > 1) {
      // Pieces of k: CTA q > 0 of the cluster stores its partial sums of this row
      // warp into the first CTA's shared memory (st.async, each store completing its
      // bytes on the first CTA's "received" barrier of the row warp) and keeps its
      // shared memory until the first CTA has them all; the first CTA adds them in
      // piece order after its own piece 0 (the same sums in the same order whatever
      // the timing) and stores the outputs.
      constexpr int kLane = xpart_lane_floats<kTwoTiles>();
      const uint32_t rank = cluster_rank();
      cluster_wait();
      // only the lanes holding tokens below m (tokens 2t, 2t + 1 and 8 + 2t, 9 + 2t)
      const bool v0 = 2 * t < m, v1 = kTwoTiles && 8 + 2 * t < m;
      if (rank != 0) {
        const uint32_t dst = map_to_rank(
            smem_u32(xpart + (((rank - 1) * kRowWarps + wr) * 32 + lane) * kLane), 0);
        const uint32_t bar = map_to_rank(xfull_bar(wr), 0);
        // timeout tests only: CTA 1 withholds its partial sums
        const bool withhold = blockIdx.x == 1 && test_withhold(status, kWithholdDecodePieces);
#pragma unroll
        for (int r = 0; r < kTiles && !withhold; ++r) {
          if (v0) st_async_f4(dst + 16 * r, make_float4(acc[r][0], acc[r][1], acc[r][2], acc[r][3]), bar);
          if (v1)
            st_async_f4(dst + 16 * (2 + r), make_float4(acc1[r][0], acc1[r][1], acc1[r][2], acc1[r][3]),
                        bar);
        }
        if (!lanes_wait(xdone_bar(wr), 0, status)) return;
        continue;  // (the end of the stream follows)
      }
      if (!lanes_wait_cluster(xfull_bar(wr), 0, status)) return;
      // every piece has landed: the other CTAs may leave (nothing to release)
      if (lane + 1 < pieces) mbar_arrive_remote_signal(map_to_rank(xdone_bar(wr), lane + 1));
      for (int q = 1; q < pieces; ++q) {
        const float4* v = reinterpret_cast<const float4*>(
            xpart + (((q - 1) * kRowWarps + wr) * 32 + lane) * kLane);
#pragma unroll
        for (int r = 0; r < kTiles; ++r) {
          if (v0) {
            const float4 a0 = v[r];
            acc[r][0] += a0.x;
            acc[r][1] += a0.y;
            acc[r][2] += a0.z;
            acc[r][3] += a0.w;
          }
          if (v1) {
            const float4 a1 = v[2 + r];
            acc1[r][0] += a1.x;
            acc1[r][1] += a1.y;
            acc1[r][2] += a1.z;
            acc1[r][3] += a1.w;
          }
        }
      }
    }
    if (kh == 0) {
      // C fragment of tile r: rows rl + 16r (slots 0, 1) and + 8 (2, 3), tokens 2t, 2t + 1
      const int n = si.n;  // rows (< 2^31) and row0 + 256 <= n + 255 fit in 32 bits
      const float post = exact ? 0.5f : 1.f;
      auto put = [&](auto* y) {
        using T = std::remove_pointer_t<decltype(y)>;
        auto store = [&](int token, int row, float v) {
          if (token < m && row < n) {
            if constexpr (std::is_same_v<T, float>)
              y[static_cast<int64_t>(token) * n + row] = post * v;
            else
              y[static_cast<int64_t>(token) * n + row] = __float2bfloat16_rn(post * v);
          }
        };
#pragma unroll
        for (int r = 0; r < kTiles; ++r) {
          const int ra = si.row0 + rl + 16 * r, rb = ra + 8;
          store(2 * t, ra, acc[r][0]);
          store(2 * t + 1, ra, acc[r][1]);
          store(2 * t, rb, acc[r][2]);
          store(2 * t + 1, rb, acc[r][3]);
          if (kTwoTiles) {
            store(8 + 2 * t, ra, acc1[r][0]);
            store(8 + 2 * t + 1, ra, acc1[r][1]);
            store(8 + 2 * t, rb, acc1[r][2]);
            store(8 + 2 * t + 1, rb, acc1[r][3]);
          }
        }
      };
      if ((si.mode >> 8) != 0)
        put(static_cast<__nv_bfloat16*>(si.y));
      else
        put(static_cast<float*>(si.y));
    }
  }
}

// Device address of g_dsched, looked up once per device.
uint32_t* dsched_base() {
  static std::atomic<uintptr_t> base[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  if (dev < 64) {
    const uintptr_t p = base[dev].load(std::memory_order_acquire);
    if (p != 0) return reinterpret_cast<uint32_t*>(p);
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_dsched) != cudaSuccess) return nullptr;
  if (dev < 64) base[dev].store(reinterpret_cast<uintptr_t>(p), std::memory_order_release);
  return static_cast<uint32_t*>(p);
}

}  // namespace

// Clusters of p CTAs of `kernel` (at `smem` bytes of shared memory each) that can
// be resident at once, asked of the runtime once per kernel, size and device.
template <typename K>
cudaError_t max_active_clusters(K* kernel, int p, int smem, int threads, int* out) {
  struct Entry {
    const void* kernel;
    int p, smem, dev, n;
  };
  static std::mutex mu;
  static Entry cache[64];
  static int used = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const void* key = reinterpret_cast<const void*>(kernel);
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (cache[i].kernel == key && cache[i].p == p && cache[i].smem == smem && cache[i].dev == dev) {
      *out = cache[i].n;
      return cudaSuccess;
    }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(p), 1, 1);
  cfg.blockDim = dim3(static_cast<unsigned>(threads), 1, 1);
  cfg.dynamicSmemBytes = static_cast<size_t>(smem);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(p);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if ((e = cudaOccupancyMaxActiveClusters(&n, kernel, &cfg)) != cudaSuccess) return e;
  if (used < 64) cache[used++] = Entry{key, p, smem, dev, n};
  *out = n;
  return cudaSuccess;
}

cudaError_t launch_decode(DecodeBatch& b, int num_sms, cudaStream_t stream) {
  static std::atomic<uint32_t> seq{0};
  // longest rows first: the units claimed last are the shortest (matrices and
  // their code maps move together; the scale maps above count stay where they are)
  int order[kDecodeMaxMats];
  for (int d = 0; d < b.count; ++d) order[d] = d;
  std::stable_sort(order, order + b.count,
                   [&](int x, int y) { return b.mats[x].k > b.mats[y].k; });
  bool sorted = true;
  for (int d = 0; d < b.count; ++d) sorted = sorted && order[d] == d;
  if (!sorted) {
    static thread_local DecodeBatch tmp;
    for (int d = 0; d < b.count; ++d) {
      tmp.mats[d] = b.mats[order[d]];
      tmp.maps[d] = b.maps[order[d]];
    }
    for (int d = 0; d < b.count; ++d) {
      b.mats[d] = tmp.mats[d];
      b.maps[d] = tmp.maps[d];
    }
  }
  int64_t blocks_of_rows = 0;
  int min_nseg = 1 << 30;
  for (int d = 0; d < b.count; ++d) {
    blocks_of_rows += (b.mats[d].n + kRows - 1) / kRows;
    const int nseg = static_cast<int>((b.mats[d].k + kSegK - 1) / kSegK);
    min_nseg = nseg < min_nseg ? nseg : min_nseg;
  }
  if (blocks_of_rows >= (int64_t{1} << 28)) return cudaErrorInvalidValue;
  if (blocks_of_rows <= 0) {
    b.total_units = 0;
    return cudaSuccess;
  }
  // scale buffers: the largest unit of scales among unit-mode matrices, a window
  // (256 rows x 32 groups, 1024-byte aligned for the swizzle) if any matrix takes
  // windows; ring slot: codes + the widest per-segment scale area + x of the m tokens
  int64_t ugroups = 0;
  int sgroups = 0;
  for (int d = 0; d < b.count; ++d) {
    const int lg = b.mats[d].log2g;
    const int64_t gpr = b.mats[d].k >> lg;
    if (b.mats[d].scale_mode == kDecodeScaleUnit) {
      const int64_t w = unit_scale_stride(static_cast<int>(gpr));  // gpr <= 32 in this mode
      ugroups = w > ugroups ? w : ugroups;
    } else if (b.mats[d].scale_mode == kDecodeScaleWin) {
      ugroups = kDecodeWinGroups;  // the most a unit-mode matrix takes too
    } else {
      const int w = seg_scale_stride(lg);
      sgroups = w > sgroups ? w : sgroups;
    }
  }
  b.ubuf_bytes = static_cast<int32_t>(kRows * ugroups * 4);
  b.scale_bytes = kRows * sgroups * 4;
  b.slot_bytes = (kCodeBytes + b.scale_bytes + b.m * kXTokBytes + 1023) & ~1023;
  const int red = b.m > 8 ? red_bytes<true>() : red_bytes<false>();
  auto smem_for = [&](int pieces, int* stages) {
    const int fixed = 1024 + kHeadBytes + red + xpart_bytes(b.m > 8, pieces) + 2 * b.ubuf_bytes;
    const int fit = (kSmemLimit - fixed) / b.slot_bytes;
    *stages = fit < kMaxStages ? fit : kMaxStages;
    return fixed + *stages * b.slot_bytes;
  };
  uint32_t* sched = dsched_base();
  if (sched == nullptr) return cudaErrorInvalidSymbol;
  sched += 2 * (seq.fetch_add(1, std::memory_order_relaxed) % kSchedSlots);
  auto go = [&](auto two, auto f16) -> cudaError_t {
    constexpr bool kTwo = decltype(two)::value, kF16 = decltype(f16)::value;
    auto* kernel = decode_kernel<kTwo, kF16, false>;
    auto* kernel_pieces = decode_kernel<kTwo, kF16, true>;
    cudaError_t err = ensure_smem_limit<decode_kernel<kTwo, kF16, false>>(kSmemLimit);
    if (err != cudaSuccess) return err;
    // Pieces of k when the blocks of rows leave SMs idle: clusters of P CTAs
    // (P = 8, 4 or 2, at most every matrix's segment count), the largest P whose
    // clusters for all the blocks are resident at once.
    int pieces = 1;
    if (blocks_of_rows < num_sms) {
      for (int p = 8; p >= 2; p >>= 1) {
        int st = 0;
        const int sm = smem_for(p, &st);
        if (p > min_nseg || st < 2 || blocks_of_rows * p > num_sms) continue;
        int nclusters = 0;
        if ((err = ensure_smem_limit<decode_kernel<kTwo, kF16, true>>(kSmemLimit)) != cudaSuccess)
          return err;
        if (max_active_clusters(kernel_pieces, p, sm, DecodeCfg<kTwo>::kThreads, &nclusters) ==
                cudaSuccess &&
            nclusters >= blocks_of_rows) {
          pieces = p;
          break;
        }
      }
    }
    b.pieces = pieces;
    int64_t units = 0;
    for (int d = 0; d < b.count; ++d) {
      b.mats[d].unit0 = static_cast<int32_t>(units);
      units += ((b.mats[d].n + kRows - 1) / kRows) * pieces;
    }
    b.total_units = static_cast<int32_t>(units);
    int stages = 0;
    const int smem = smem_for(pieces, &stages);
    b.stages = stages;
    if (b.stages < 2) return cudaErrorInvalidValue;
    // Every decode launch may start before the previous launch on the stream has
    // completed (programmatic serialisation): its CTAs set up and prefetch into L2,
    // then wait for that grid before reading or writing anything it might touch.
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(DecodeCfg<kTwo>::kThreads, 1, 1);
    cfg.dynamicSmemBytes = static_cast<size_t>(smem);
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    if (pieces == 1) {
      // persistent: one CTA per SM at most, units claimed from the scheduler
      cfg.gridDim = dim3(static_cast<unsigned>(units < num_sms ? units : num_sms), 1, 1);
      cfg.numAttrs = 1;
      return cudaLaunchKernelEx(&cfg, kernel, b, sched);
    }
    // one CTA per unit, clusters of `pieces` CTAs over one block of rows
    cfg.gridDim = dim3(static_cast<unsigned>(units), 1, 1);
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = static_cast<unsigned>(pieces);
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kernel_pieces, b, sched);
  };
  cudaError_t e;
  if (b.m > 8)
    e = b.in_f16 ? go(std::true_type{}, std::true_type{}) : go(std::true_type{}, std::false_type{});
  else
    e = b.in_f16 ? go(std::false_type{}, std::true_type{}) : go(std::false_type{}, std::false_type{});
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace tq
