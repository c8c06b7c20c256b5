// quantize.cu — §3.1 quantiser: per-group absmean scale, ternary codes, 2-bit packing,
// zero count per group. One pass over the fp32 latent weights; HBM-bound.
//
// The weight matrix is treated as one flat array: groups (g | k) and code words
// (16 | k) never straddle a row, so group j of row n is flat group n*(k/g)+j and
// the outputs are flat arrays too.
//
// Streaming: a persistent grid (two CTAs per SM) splits the flat array into
// stages of 8192 weights (32 KB), claimed one at a time from a per-launch atomic
// counter (SMs do not all receive HBM data at the same rate; static equal shares
// left the slowest CTA ~40% behind). One producer thread keeps a ring of kStages
// stages in flight with
// cp.async.bulk (L2 evict-first: the latent weights are read once), so the
// loads never wait for the arithmetic; sixteen consumer warps split every stage,
// 512 weights each, and release the slot through an "empty" mbarrier. Two CTAs
// per SM keep 32 blocks of 512 weights in process per SM, which the per-block
// latency (shuffle chain, reductions) needs to keep pace with HBM.
//
// Consumer: each lane owns 16 consecutive weights — one code word. A group
// spans g/16 consecutive lanes; its |w| sum and its zero count are reduced with
// log2(g/16) xor-shuffles each (the zero count of a word is 16 - popc(word &
// 0x5555...) because every non-zero code has its low bit set; a redux.sync over
// the group's lanes, whose mask differs between the groups of a warp, was issued
// once per group: 16 times per warp at g = 32).
//
// Code decision: see quant_code.cuh.
//
// Fused variant (tq_quantize_with_transpose): the same stages, then, in the same
// cooperative launch, a grid barrier (a counter per launch slot, bounded wait, reset
// by the last CTA past it) and the whole grid transposes the codes into codes_t,
// reading them back through L2 (16 x 16 blocks, transpose_block16).
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"
#include "ptx.cuh"
#include "quant_code.cuh"

namespace tq {
namespace {

constexpr int kUnit = 512;                      // weights per consumer warp per stage
constexpr int kConsumers = 16;                  // consumer warps
constexpr int kThreads = (kConsumers + 1) * 32; // + one producer warp
constexpr int kStageW = kConsumers * kUnit;     // 8192 weights per stage
constexpr int kStageBytes = kStageW * 4;        // 32 KB
constexpr int kStages = 3;                      // per CTA; two CTAs per SM
constexpr int kCtasPerSm = 2;
constexpr int kSmemBytes = kStages * kStageBytes + 2 * kStages * 8 + 128;

// Stage scheduler of one launch: {next dynamic stage, CTAs done}. Zero at the
// start of a launch; the last CTA to finish claiming puts both back to zero.
// Launches take the slots in turn, so up to kSchedSlots launches may be in
// flight at once.
constexpr int kSchedSlots = 256;
__device__ uint32_t g_sched[kSchedSlots][2];
// Grid barrier of the fused quantize + transpose, per launch slot: {arrived, passed}.
__device__ uint32_t g_tbar[kSchedSlots][2];

// Matrix d of a batch owns the global stages [stage0, stage0 + ceil(total / kStageW));
// a stage never spans two matrices (a matrix's last stage may be short).
__device__ __forceinline__ int find_stage_mat(const QuantMat* mats, int count, int64_t st) {
  int lo = 0, hi = count - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (mats[mid].stage0 <= st) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// codes [n][k/16] -> codes_t [k][ldt]. Each thread owns one 16 x 16 block of 2-bit
// codes (16 rows n of one code word c) and transposes it in registers with four
// levels of block swaps (8, 4, 2, 1 fields; the two byte-sized levels are byte
// permutes). Field p of a word holds element i(p) = 2 (p % 8) + p / 8 (the packing
// puts the even elements in the low half), so the rows are loaded in the order
// i(q) and the transposed word p is stored as output row i(p): the plain
// transpose then lands every element at its packed position. Rows past n read as
// 0, which writes the zero padding of the last words. The codes are read through
// L2 (ld.global.cg): in the fused quantize they were written by the same launch.
__device__ __forceinline__ void swap_fields(uint32_t& a, uint32_t& c, int shift, uint32_t mask) {
  const uint32_t t = ((a >> shift) ^ c) & mask;
  c ^= t;
  a ^= t << shift;
}

__device__ __forceinline__ void transpose_block16(const uint32_t* codes, int64_t n, int64_t words,
                                                  uint32_t* codes_t, int64_t ldt, int64_t c,
                                                  int64_t r16) {
  uint32_t t[16];
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    const int64_t row = 16 * r16 + 2 * (q & 7) + (q >> 3);
    t[q] = row < n ? __ldcg(codes + row * words + c) : 0u;
  }
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    const uint32_t a = t[w], b = t[w + 8];
    t[w] = __byte_perm(a, b, 0x5410);
    t[w + 8] = __byte_perm(a, b, 0x7632);
  }
#pragma unroll
  for (int w = 0; w < 16; ++w) {
    if (w & 4) continue;
    const uint32_t a = t[w], b = t[w + 4];
    t[w] = __byte_perm(a, b, 0x6240);
    t[w + 4] = __byte_perm(a, b, 0x7351);
  }
#pragma unroll
  for (int w = 0; w < 16; ++w)
    if (!(w & 2)) swap_fields(t[w], t[w + 2], 4, 0x0F0F0F0Fu);
#pragma unroll
  for (int w = 0; w < 16; ++w)
    if (!(w & 1)) swap_fields(t[w], t[w + 1], 2, 0x33333333u);
  uint32_t* out = codes_t + 16 * c * ldt + r16;
#pragma unroll
  for (int p = 0; p < 16; ++p) out[(2 * (p & 7) + (p >> 3)) * ldt] = t[p];
}

// A warp transposes 8 consecutive words x 4 consecutive 16-row groups (32-byte
// reads, 16-byte writes): tile `tile` of a grid of ceil(words / 8) tiles per row
// of 4 groups.
__device__ __forceinline__ void transpose_warp_tile(const uint32_t* codes, int64_t n, int64_t words,
                                                    uint32_t* codes_t, int64_t ldt, int64_t tile,
                                                    int lane) {
  const int64_t tc = (words + 7) / 8;
  const int64_t c = (tile % tc) * 8 + (lane & 7);
  const int64_t r16 = (tile / tc) * 4 + (lane >> 3);
  if (c < words && r16 < ldt) transpose_block16(codes, n, words, codes_t, ldt, c, r16);
}

// The transposed-codes output of the fused quantize (tq_quantize_with_transpose).
struct QuantT {
  uint32_t* codes_t;  // [k][ldt]
  int64_t n, words, ldt;
  uint32_t* bar;      // grid barrier of the launch: {arrived, passed}
};

template <int G, int kMax, bool kGiven, bool kT>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    quantize_kernel(const __grid_constant__ QuantBatch<kMax> b, uint32_t* sched, int* status,
                    const QuantT tt) {
  static_assert(G == 32 || G == 64 || G == 128 || G == 256 || G == 512, "group size");
  static_assert(kStageW % G == 0, "a group never straddles a stage");
  constexpr int kLanesPerGroup = G / 16;
  constexpr float kInvG = 1.0f / G;  // exact: G is a power of two
  extern __shared__ uint8_t smem_raw[];
  __shared__ int64_t stage_of[kStages];  // local stage held by each slot; -1: end of stream
  __shared__ int mat_of[kStages];        // its matrix
  uint8_t* smem = align_shared<128>(smem_raw);
  const uint32_t ring = smem_u32(smem);
  const uint32_t bars = ring + kStages * kStageBytes;
  auto full_bar = [&](int s) { return bars + 8 * s; };
  auto empty_bar = [&](int s) { return bars + 8 * (kStages + s); };

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t nstages = b.nstages;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), kConsumers);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kConsumers) {
    // ------------------------------------------------------------ producer
    // The first ring's worth of stages is dealt round-robin (no claim latency
    // before the first loads); later stages are claimed one at a time from the
    // launch's counter, so SMs that receive their data faster take more of them
    // and all CTAs end together.
    if (lane == 0) {
      const uint64_t policy = policy_evict_first();
      const int64_t dealt = static_cast<int64_t>(kStages) * gridDim.x;
      int round0 = 0;
      auto claim = [&]() -> int64_t {
        if (round0 < kStages) return blockIdx.x + static_cast<int64_t>(round0++) * gridDim.x;
        return dealt + atomicAdd(&sched[0], 1u);
      };
      int slot = 0;
      uint32_t parity = 0;  // phase parity of the slot's current round
      int64_t issued = 0;
      bool ok = true;
      int64_t st = claim();
      for (;;) {
        if (issued >= kStages && !mbar_wait(empty_bar(slot), parity ^ 1u, status)) {
          ok = false;
          break;
        }
        if (st >= nstages) {  // end of the stream: an empty stage tells the consumers
          stage_of[slot] = -1;
          mbar_arrive(full_bar(slot));
          break;
        }
        const int d = kMax == 1 ? 0 : find_stage_mat(b.mats, b.count, st);
        const QuantMat& mt = b.mats[d];
        const int64_t ls = st - mt.stage0;
        const int64_t e0 = ls * kStageW;
        const int64_t cnt = mt.total - e0 < kStageW ? mt.total - e0 : kStageW;
        const uint32_t bytes = static_cast<uint32_t>(cnt) * 4u;
        stage_of[slot] = ls;
        mat_of[slot] = d;
        mbar_arrive_expect_tx(full_bar(slot), bytes);
        bulk_load(ring + slot * kStageBytes, mt.w + e0, bytes, full_bar(slot), policy);
        st = claim();  // a counter claim is in flight during the wait above
        ++issued;
        if (++slot == kStages) {
          slot = 0;
          parity ^= 1u;
        }
      }
      // this CTA claims no more: the last CTA to get here resets the scheduler
      __threadfence();
      if (atomicAdd(&sched[1], 1u) == gridDim.x - 1) {
        atomicExch(&sched[0], 0u);
        atomicExch(&sched[1], 0u);
      }
      // Nothing may still write this CTA's ring when it exits. Normally the
      // consumers have waited for every stage before they see the end marker;
      // if they gave up, wait here for the stages issued last (a slot's newest
      // phase is its last load: no end marker was written on this path).
      if (!ok) {
        for (int64_t j = issued > kStages ? issued - kStages : 0; j < issued; ++j) {
          if (!mbar_wait(full_bar(static_cast<int>(j % kStages)),
                         static_cast<uint32_t>((j / kStages) & 1), status))
            break;
        }
      }
    }
    if constexpr (!kT) return;
  } else {
    // ------------------------------------------------------------ consumers
    // (a lambda: its returns end this warp's stages, not the kernel)
    [&] {
      int slot = 0;
      uint32_t parity = 0;
      // timeout tests only: this warp withholds its first "empty" arrival
      bool withhold = blockIdx.x == 0 && warp == 0 && test_withhold(status, kWithholdQuantizeEmpty);
      for (;;) {
        if (!lanes_wait(full_bar(slot), parity, status)) return;
        const int64_t ls = stage_of[slot];
        if (ls < 0) return;
        const QuantMat& mt = b.mats[kMax == 1 ? 0 : mat_of[slot]];
        const int64_t total = mt.total;
        const int64_t base = ls * kStageW + warp * kUnit;
        const int64_t e = base + lane * 16;
        if (e < total) {
          // lanes of this block that hold weights; a multiple of g/16 (g | total)
          const int64_t rem = total - base;
          const unsigned live = rem >= kUnit ? 0xffffffffu : (1u << (rem >> 4)) - 1u;
          const float4* src = reinterpret_cast<const float4*>(smem + slot * kStageBytes +
                                                              (warp * kUnit + lane * 16) * 4);
          float4 v[4];
    #pragma unroll
          for (int j = 0; j < 4; ++j) v[j] = src[j];
          const float x[16] = {v[0].x, v[0].y, v[0].z, v[0].w, v[1].x, v[1].y, v[1].z, v[1].w,
                               v[2].x, v[2].y, v[2].z, v[2].w, v[3].x, v[3].y, v[3].z, v[3].w};
          float s = 0.f;
          uint32_t word;
          if constexpr (kGiven) {
            // the learnable-scale variant: the caller's scale decides, of either sign
            word = code_word_any(x, __ldg(mt.given_scale + e / G), live);
          } else {
            float sum = 0.f;
    #pragma unroll
            for (int j = 0; j < 4; ++j)
              sum += (fabsf(v[j].x) + fabsf(v[j].y)) + (fabsf(v[j].z) + fabsf(v[j].w));
    #pragma unroll
            for (int off = 1; off < kLanesPerGroup; off <<= 1) sum += __shfl_xor_sync(live, sum, off);
            s = sum * kInvG;  // s = (1/g) * sum |w|
            // the decoupled quantizer decides against tau = f_row * s (one fp32 product)
            const float tau = mt.row_factor == nullptr ? s : __fmul_rn(s, mt.row_factor[e / mt.k]);
            // thresholds below 2^-100 (all-zero or denormal groups) take the division
            const bool tiny = tau < 0x1p-100f;
            word = __any_sync(live, tiny)
                       ? (tiny ? code_word<true>(x, tau) : code_word<false>(x, tau))
                       : code_word<false>(x, tau);
          }
          // zero count of the group: xor-shuffles over its lanes (a redux.sync whose
          // mask differs between the groups of a warp is issued once per group)
          unsigned zs = 16u - static_cast<unsigned>(__popc(word & 0x55555555u));
          if constexpr (kLanesPerGroup == 32) {
            zs = __reduce_add_sync(live, zs);
          } else {
          #pragma unroll
            for (int off = 1; off < kLanesPerGroup; off <<= 1) zs += __shfl_xor_sync(live, zs, off);
          }
          const int zc = static_cast<int>(zs);
          mt.codes[e >> 4] = word;
          if ((lane & (kLanesPerGroup - 1)) == 0) {
            if (!kGiven) mt.scales[e / G] = s;
            mt.zeros[e / G] = zc;
          }
        }
        __syncwarp();
        if (lane == 0 && !withhold) mbar_arrive(empty_bar(slot));
        withhold = false;
        if (++slot == kStages) {
          slot = 0;
          parity ^= 1u;
        }
      }
    }();
    if constexpr (!kT) return;
  }

  if constexpr (kT) {
    // Transposed codes (fused tq_codes_transpose): once every CTA has stored its
    // stages' codes, the grid transposes them while they are still in L2. The
    // launch is cooperative, so all CTAs are resident and the barrier completes;
    // if it gives up, the status says so and the transpose is skipped.
    __shared__ int passed;
    __syncthreads();  // this CTA's code stores precede its arrival
    if (threadIdx.x == 0) {
      __threadfence();
      atomicAdd(&tt.bar[0], 1u);
      passed = counter_wait(&tt.bar[0], gridDim.x, status) ? 1 : 0;
      // the last CTA past the barrier resets it for the next launch on this slot
      if (atomicAdd(&tt.bar[1], 1u) == gridDim.x - 1) {
        atomicExch(&tt.bar[0], 0u);
        atomicExch(&tt.bar[1], 0u);
      }
    }
    __syncthreads();
    if (passed != 0) {
      const int64_t tiles = ((tt.words + 7) / 8) * ((tt.ldt + 3) / 4);
      const int64_t warps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
      // tiles dealt across the CTAs first (tile = warp * grid + CTA), so that every SM
      // takes a share of the ~2000 tiles: dealt CTA by CTA, the first ~125 CTAs took
      // them all (2 us more of the launch's 28.7 after a 70 MB dirty write)
      for (int64_t tile = static_cast<int64_t>(warp) * gridDim.x + blockIdx.x; tile < tiles;
           tile += warps)
        transpose_warp_tile(b.mats[0].codes, tt.n, tt.words, tt.codes_t, tt.ldt, tile, lane);
    }
  }
}

// codes [n][k/16] -> codes_t [k][ldt], one warp per tile of 8 words x 4 groups of 16 rows.
__global__ void __launch_bounds__(256) transpose_codes_kernel(const uint32_t* __restrict__ codes,
                                                              int64_t n, int64_t words,
                                                              uint32_t* __restrict__ codes_t,
                                                              int64_t ldt, int64_t tiles) {
  const int64_t tile = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  if (tile < tiles) transpose_warp_tile(codes, n, words, codes_t, ldt, tile, threadIdx.x & 31);
}

// Device address of g_sched, looked up once per device.
uint32_t* sched_base() {
  static std::atomic<uintptr_t> base[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  if (dev < 64) {
    const uintptr_t p = base[dev].load(std::memory_order_acquire);
    if (p != 0) return reinterpret_cast<uint32_t*>(p);
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_sched) != cudaSuccess) return nullptr;
  if (dev < 64) base[dev].store(reinterpret_cast<uintptr_t>(p), std::memory_order_release);
  return static_cast<uint32_t*>(p);
}

// Device address of g_tbar, looked up once per device.
uint32_t* tbar_base() {
  static std::atomic<uintptr_t> base[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  if (dev < 64) {
    const uintptr_t p = base[dev].load(std::memory_order_acquire);
    if (p != 0) return reinterpret_cast<uint32_t*>(p);
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_tbar) != cudaSuccess) return nullptr;
  if (dev < 64) base[dev].store(reinterpret_cast<uintptr_t>(p), std::memory_order_release);
  return static_cast<uint32_t*>(p);
}

std::atomic<uint32_t> g_seq{0};  // launch slot of the scheduler and the grid barrier

// t.codes_t != null: the fused quantize + transpose, a cooperative launch of at
// most the CTAs that fit on the device at once.
template <int G, int kMax, bool kGiven, bool kT>
cudaError_t launch(const QuantBatch<kMax>& b, int* status, int num_sms, cudaStream_t stream,
                   QuantT t = QuantT{}) {
  if (b.nstages <= 0) return cudaSuccess;
  if (b.nstages >= (int64_t{1} << 31)) return cudaErrorInvalidValue;
  auto kern = quantize_kernel<G, kMax, kGiven, kT>;
  cudaError_t e = ensure_smem_limit<quantize_kernel<G, kMax, kGiven, kT>>(kSmemBytes);
  if (e != cudaSuccess) return e;
  int per_sm = kCtasPerSm;
  if (kT) {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, kSmemBytes);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorCooperativeLaunchTooLarge;
    if (per_sm > kCtasPerSm) per_sm = kCtasPerSm;
  }
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  const int64_t blocks = b.nstages < cap ? b.nstages : cap;
  uint32_t* sched = sched_base();
  uint32_t* tbar = tbar_base();
  if (sched == nullptr || tbar == nullptr) return cudaErrorInvalidSymbol;
  const uint32_t slot = g_seq.fetch_add(1, std::memory_order_relaxed) % kSchedSlots;
  sched += 2 * slot;
  if (!kT) {
    kern<<<static_cast<unsigned>(blocks), kThreads, kSmemBytes, stream>>>(b, sched, status, t);
    return cudaGetLastError();
  }
  t.bar = tbar + 2 * slot;
  void* args[] = {const_cast<QuantBatch<kMax>*>(&b), &sched, &status, &t};
  return cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(kern),
                                     dim3(static_cast<unsigned>(blocks)), dim3(kThreads), args,
                                     kSmemBytes, stream);
}

template <int kMax, bool kGiven, bool kT = false>
cudaError_t launch_g(const QuantBatch<kMax>& b, int g, int* status, int num_sms,
                     cudaStream_t stream, QuantT t = QuantT{}) {
  switch (g) {
    case 32: return launch<32, kMax, kGiven, kT>(b, status, num_sms, stream, t);
    case 64: return launch<64, kMax, kGiven, kT>(b, status, num_sms, stream, t);
    case 128: return launch<128, kMax, kGiven, kT>(b, status, num_sms, stream, t);
    case 256: return launch<256, kMax, kGiven, kT>(b, status, num_sms, stream, t);
    case 512: return launch<512, kMax, kGiven, kT>(b, status, num_sms, stream, t);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

namespace {

// Magnitude gradient of the decoupled quantizer: dalpha_g = sum over the group of
// dW * c. A lane takes one code word (16 weights, its dW as four float4) and adds
// the dW of its non-zero codes with their signs, in weight order; the g/16 lanes
// of a group then add their sums with xor-shuffles (groups lie within one warp's
// 32 words, and a warp holds whole groups). Plain vector loads: a secondary pass.
template <int G>
__global__ void __launch_bounds__(256) alpha_grad_kernel(const float* __restrict__ dw,
                                                         const uint32_t* __restrict__ codes,
                                                         int64_t words, float* __restrict__ dalpha) {
  constexpr int kLanesPerGroup = G / 16;
  const int lane = threadIdx.x & 31;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31);
       base < words; base += stride) {
    const int64_t wi = base + lane;
    if (wi >= words) continue;  // whole groups: the lanes of a group agree
    const uint32_t c = __ldg(codes + wi);
    const float4* p = reinterpret_cast<const float4*>(dw + wi * 16);
    float sum = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 v4 = __ldg(p + q);
      const float v[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int j = 4 * q + i;
        const int bit = 16 * (j & 1) + 2 * (j >> 1);  // code j of the word (include/tq.h)
        const float t = (c >> (bit + 1)) & 1u ? -v[i] : v[i];
        sum += (c >> bit) & 1u ? t : 0.f;
      }
    }
    const unsigned gmask =
        kLanesPerGroup == 32 ? 0xffffffffu
                             : ((1u << kLanesPerGroup) - 1u) << (lane & ~(kLanesPerGroup - 1));
#pragma unroll
    for (int off = 1; off < kLanesPerGroup; off <<= 1) sum += __shfl_xor_sync(gmask, sum, off);
    if ((lane & (kLanesPerGroup - 1)) == 0) dalpha[wi / kLanesPerGroup] = sum;
  }
}

template <int G>
cudaError_t launch_ag(const float* dw, const uint32_t* codes, int64_t words, float* dalpha,
                      int num_sms, cudaStream_t stream) {
  const int64_t need = (words + 255) / 256;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  alpha_grad_kernel<G><<<static_cast<unsigned>(need < cap ? need : cap), 256, 0, stream>>>(
      dw, codes, words, dalpha);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_alpha_grad(const float* dw, const uint32_t* codes, int64_t n, int64_t k, int g,
                              float* dalpha, int num_sms, cudaStream_t stream) {
  const int64_t words = n * k / 16;
  if (words <= 0) return cudaSuccess;
  switch (g) {
    case 32: return launch_ag<32>(dw, codes, words, dalpha, num_sms, stream);
    case 64: return launch_ag<64>(dw, codes, words, dalpha, num_sms, stream);
    case 128: return launch_ag<128>(dw, codes, words, dalpha, num_sms, stream);
    case 256: return launch_ag<256>(dw, codes, words, dalpha, num_sms, stream);
    case 512: return launch_ag<512>(dw, codes, words, dalpha, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

namespace {

// dscale of the learnable-scale variant: a lane per code word; per group the sums
// A = sum dw * c and B = sum over |w| < |s| of dw * w, reduced over the group's
// lanes; dscale = A - B / s (B is 0 when s is 0: no |w| is below it).
template <int G>
__global__ void __launch_bounds__(256) scale_grad_kernel(const float* __restrict__ w,
                                                         const float* __restrict__ dw,
                                                         const uint32_t* __restrict__ codes,
                                                         const float* __restrict__ scales,
                                                         int64_t words, float* __restrict__ ds) {
  constexpr int kLanesPerGroup = G / 16;
  const int lane = threadIdx.x & 31;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31);
       base < words; base += stride) {
    const int64_t wi = base + lane;
    if (wi >= words) continue;  // whole groups: the lanes of a group agree
    const int64_t gi = wi / kLanesPerGroup;
    const uint32_t c = __ldg(codes + wi);
    const float s = __ldg(scales + gi);
    const float as = fabsf(s);
    const float4* pd = reinterpret_cast<const float4*>(dw + wi * 16);
    const float4* pw = reinterpret_cast<const float4*>(w + wi * 16);
    float a = 0.f, b = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 d4 = __ldg(pd + q);
      const float4 w4 = __ldg(pw + q);
      const float d[4] = {d4.x, d4.y, d4.z, d4.w};
      const float x[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int j = 4 * q + i;
        const int bit = 16 * (j & 1) + 2 * (j >> 1);  // code j of the word (include/tq.h)
        const float t = (c >> (bit + 1)) & 1u ? -d[i] : d[i];
        a += (c >> bit) & 1u ? t : 0.f;
        b += fabsf(x[i]) < as ? d[i] * x[i] : 0.f;
      }
    }
    const unsigned gmask =
        kLanesPerGroup == 32 ? 0xffffffffu
                             : ((1u << kLanesPerGroup) - 1u) << (lane & ~(kLanesPerGroup - 1));
#pragma unroll
    for (int off = 1; off < kLanesPerGroup; off <<= 1) {
      a += __shfl_xor_sync(gmask, a, off);
      b += __shfl_xor_sync(gmask, b, off);
    }
    if ((lane & (kLanesPerGroup - 1)) == 0) ds[gi] = b == 0.f ? a : a - __fdiv_rn(b, s);
  }
}

template <int G>
cudaError_t launch_sg(const float* w, const float* dw, const uint32_t* codes, const float* scales,
                      int64_t words, float* ds, int num_sms, cudaStream_t stream) {
  const int64_t need = (words + 255) / 256;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  scale_grad_kernel<G><<<static_cast<unsigned>(need < cap ? need : cap), 256, 0, stream>>>(
      w, dw, codes, scales, words, ds);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_scale_grad(const float* w, const float* dw, const uint32_t* codes,
                              const float* scales, int64_t n, int64_t k, int g, float* dscale,
                              int num_sms, cudaStream_t stream) {
  const int64_t words = n * k / 16;
  if (words <= 0) return cudaSuccess;
  switch (g) {
    case 32: return launch_sg<32>(w, dw, codes, scales, words, dscale, num_sms, stream);
    case 64: return launch_sg<64>(w, dw, codes, scales, words, dscale, num_sms, stream);
    case 128: return launch_sg<128>(w, dw, codes, scales, words, dscale, num_sms, stream);
    case 256: return launch_sg<256>(w, dw, codes, scales, words, dscale, num_sms, stream);
    case 512: return launch_sg<512>(w, dw, codes, scales, words, dscale, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_transpose_codes(const uint32_t* codes, int64_t n, int64_t k, uint32_t* codes_t,
                                   cudaStream_t stream) {
  const int64_t ldt = 4 * ((n + 63) / 64), words = k / 16;
  const int64_t tiles = ((words + 7) / 8) * ((ldt + 3) / 4);
  transpose_codes_kernel<<<static_cast<unsigned>((tiles + 7) / 8), 256, 0, stream>>>(
      codes, n, words, codes_t, ldt, tiles);
  return cudaGetLastError();
}

cudaError_t launch_quantize(const float* w, int64_t n, int64_t k, int g, uint32_t* codes,
                            float* scales, int32_t* zeros, int* status, int num_sms,
                            cudaStream_t stream, const float* row_factor,
                            const float* given_scale) {
  QuantBatch<1> b{};
  b.mats[0] = QuantMat{w, codes, scales, zeros, n * k, 0, row_factor, k, given_scale};
  b.count = 1;
  b.nstages = (n * k + kStageW - 1) / kStageW;
  return given_scale != nullptr ? launch_g<1, true>(b, g, status, num_sms, stream)
                                 : launch_g<1, false>(b, g, status, num_sms, stream);
}

cudaError_t launch_quantize_t(const float* w, int64_t n, int64_t k, int g, uint32_t* codes,
                              float* scales, int32_t* zeros, uint32_t* codes_t, int* status,
                              int num_sms, cudaStream_t stream) {
  QuantBatch<1> b{};
  b.mats[0] = QuantMat{w, codes, scales, zeros, n * k, 0, nullptr, k, nullptr};
  b.count = 1;
  b.nstages = (n * k + kStageW - 1) / kStageW;
  const QuantT t{codes_t, n, k / 16, 4 * ((n + 63) / 64), nullptr};
  return launch_g<1, false, true>(b, g, status, num_sms, stream, t);
}

cudaError_t launch_quantize_batched(QuantBatch<kQuantMaxMats>& b, int g, int* status,
                                    int num_sms, cudaStream_t stream) {
  int64_t st = 0;
  for (int d = 0; d < b.count; ++d) {
    b.mats[d].stage0 = st;
    st += (b.mats[d].total + kStageW - 1) / kStageW;
  }
  b.nstages = st;
  return launch_g<kQuantMaxMats, false>(b, g, status, num_sms, stream);
}

}  // namespace tq
