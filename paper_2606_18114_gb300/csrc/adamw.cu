// adamw.cu — the optimizer step of the latent weights fused with their
// requantization (§3.3: AdamW on the fp32 latent weights; §3.1: the group scales
// and ternary codes are recomputed from the weights every step). One pass reads
// W, dW, m and v (16 B per weight) and writes W, m, v (12 B) and the codes,
// scales and zero counts of the new W (0.25 + 8/g B), instead of an optimizer pass
// followed by a quantize pass that reads W again. HBM-bound.
//
// Streaming as in the quantize kernel: the matrix is one flat array (groups and
// code words never straddle a row); stages of 4096 weights — 64 KB over the four
// inputs — are dealt round-robin for the first ring and then claimed from a
// per-launch counter; one producer thread keeps a ring of three stages in flight
// with cp.async.bulk (L2 evict-first: every input is read once); eight consumer
// warps split each stage, 512 weights a warp, 16 a lane.
//
// Update (every operation one IEEE fp32 operation, in this order, no fused
// multiply-add: the oracle reproduces it bit for bit):
//   g' = g * grad_scale
//   m  = b1 * m + (1 - b1) * g'
//   v  = b2 * v + (1 - b2) * (g' * g')
//   w  = w * (1 - lr * wd) - step_size * (m / (sqrt(v) * inv_bc2_sqrt + eps))
// with step_size = lr / (1 - b1^t) and inv_bc2_sqrt = 1 / sqrt(1 - b2^t), the step
// constants computed on the host in fp64 and rounded once to fp32. The new W is
// then quantized exactly as tq_quantize does (quant_code.cuh), or against
// caller-given scales (the learnable-scale variant), or not at all (a plain AdamW
// step over any fp32 array of a multiple of 16 elements, e.g. those scales).
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "kernels.cuh"
#include "ptx.cuh"
#include "quant_code.cuh"

namespace tq {
namespace {

constexpr int kUnit = 512;                         // weights per consumer warp per stage
constexpr int kConsumers = 8;
constexpr int kThreads = (kConsumers + 1) * 32;   // + one producer warp
constexpr int kStageW = kConsumers * kUnit;       // 4096 weights per stage
constexpr int kArrayBytes = kStageW * 4;          // 16 KB per input array
constexpr int kStageBytes = 4 * kArrayBytes;      // w, g, m, v
constexpr int kStages = 3;
constexpr int kSmemBytes = kStages * kStageBytes + 2 * kStages * 8 + 128;

constexpr int kSchedSlots = 256;
__device__ uint32_t g_asched[kSchedSlots][2];  // {next dynamic stage, CTAs done} per launch

__device__ __forceinline__ float4 ld4(const uint8_t* p) { return *reinterpret_cast<const float4*>(p); }

// kMode: what follows the update — the absmean requantization (kAbsmean), codes
// against the caller's scales (kGivenScales), or nothing (kPlain).
enum : int { kAbsmean = 0, kGivenScales = 1, kPlain = 2 };

template <int G, int kMode>
__global__ void __launch_bounds__(kThreads, 1)
    adamw_requantize_kernel(const AdamwArgs a, uint32_t* sched, int* status) {
  constexpr int kLanesPerGroup = G / 16;
  constexpr float kInvG = 1.0f / G;
  extern __shared__ uint8_t smem_raw[];
  __shared__ int64_t stage_of[kStages];  // stage held by each slot; -1: end of stream
  uint8_t* smem = align_shared<128>(smem_raw);
  const uint32_t ring = smem_u32(smem);
  const uint32_t bars = ring + kStages * kStageBytes;
  auto full_bar = [&](int s) { return bars + 8 * s; };
  auto empty_bar = [&](int s) { return bars + 8 * (kStages + s); };
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t total = a.total;
  const int64_t nstages = (total + kStageW - 1) / kStageW;

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
    if (lane == 0) {
      const uint64_t policy = policy_evict_first();
      const int64_t dealt = static_cast<int64_t>(kStages) * gridDim.x;
      int round0 = 0;
      auto claim = [&]() -> int64_t {
        if (round0 < kStages) return blockIdx.x + static_cast<int64_t>(round0++) * gridDim.x;
        return dealt + atomicAdd(&sched[0], 1u);
      };
      int slot = 0;
      uint32_t parity = 0;
      int64_t issued = 0;
      bool ok = true;
      int64_t st = claim();
      for (;;) {
        if (issued >= kStages && !mbar_wait(empty_bar(slot), parity ^ 1u, status)) {
          ok = false;
          break;
        }
        if (st >= nstages) {  // end of the stream
          stage_of[slot] = -1;
          mbar_arrive(full_bar(slot));
          break;
        }
        const int64_t e0 = st * kStageW;
        const int64_t cnt = total - e0 < kStageW ? total - e0 : kStageW;
        const uint32_t bytes = static_cast<uint32_t>(cnt) * 4u;  // a multiple of 64 (16 | total)
        const uint32_t dst = ring + slot * kStageBytes;
        stage_of[slot] = st;
        mbar_arrive_expect_tx(full_bar(slot), 4 * bytes);
        bulk_load(dst, a.w + e0, bytes, full_bar(slot), policy);
        bulk_load(dst + kArrayBytes, a.grad + e0, bytes, full_bar(slot), policy);
        bulk_load(dst + 2 * kArrayBytes, a.m + e0, bytes, full_bar(slot), policy);
        bulk_load(dst + 3 * kArrayBytes, a.v + e0, bytes, full_bar(slot), policy);
        st = claim();
        ++issued;
        if (++slot == kStages) {
          slot = 0;
          parity ^= 1u;
        }
      }
      __threadfence();
      if (atomicAdd(&sched[1], 1u) == gridDim.x - 1) {  // the last CTA resets the scheduler
        atomicExch(&sched[0], 0u);
        atomicExch(&sched[1], 0u);
      }
      if (!ok) {  // nothing may still write the ring when the CTA exits
        for (int64_t j = issued > kStages ? issued - kStages : 0; j < issued; ++j)
          if (!mbar_wait(full_bar(static_cast<int>(j % kStages)),
                         static_cast<uint32_t>((j / kStages) & 1), status))
            break;
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const AdamwConst c = a.c;
  int slot = 0;
  uint32_t parity = 0;
  for (;;) {
    if (!lanes_wait(full_bar(slot), parity, status)) return;
    const int64_t st = stage_of[slot];
    if (st < 0) return;
    const int64_t base = st * kStageW + warp * kUnit;
    const int64_t e = base + lane * 16;
    if (e < total) {
      const int64_t rem = total - base;
      const unsigned live = rem >= kUnit ? 0xffffffffu : (1u << (rem >> 4)) - 1u;
      const uint8_t* src = smem + slot * kStageBytes + (warp * kUnit + lane * 16) * 4;
      float x[16];
      float mo[16], vo[16];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float4 w4 = ld4(src + 16 * q);
        const float4 g4 = ld4(src + kArrayBytes + 16 * q);
        const float4 m4 = ld4(src + 2 * kArrayBytes + 16 * q);
        const float4 v4 = ld4(src + 3 * kArrayBytes + 16 * q);
        const float wi[4] = {w4.x, w4.y, w4.z, w4.w}, gi[4] = {g4.x, g4.y, g4.z, g4.w};
        const float mi[4] = {m4.x, m4.y, m4.z, m4.w}, vi[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float gg = __fmul_rn(gi[i], c.grad_scale);
          const float m1 = __fadd_rn(__fmul_rn(c.b1, mi[i]), __fmul_rn(c.omb1, gg));
          const float v1 = __fadd_rn(__fmul_rn(c.b2, vi[i]), __fmul_rn(c.omb2, __fmul_rn(gg, gg)));
          const float den = __fadd_rn(__fmul_rn(__fsqrt_rn(v1), c.inv_bc2_sqrt), c.eps);
          x[4 * q + i] = __fsub_rn(__fmul_rn(wi[i], c.decay), __fmul_rn(c.step_size, __fdiv_rn(m1, den)));
          mo[4 * q + i] = m1;
          vo[4 * q + i] = v1;
        }
      }
      float4* wd = reinterpret_cast<float4*>(a.w + e);
      float4* md = reinterpret_cast<float4*>(a.m + e);
      float4* vd = reinterpret_cast<float4*>(a.v + e);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        wd[q] = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
        md[q] = make_float4(mo[4 * q], mo[4 * q + 1], mo[4 * q + 2], mo[4 * q + 3]);
        vd[q] = make_float4(vo[4 * q], vo[4 * q + 1], vo[4 * q + 2], vo[4 * q + 3]);
      }
      if constexpr (kMode != kPlain) {
        // requantize the new weights: against their absmean (as tq_quantize) or
        // against the caller's scales (the learnable-scale variant)
        float s = 0.f;
        uint32_t word;
        if constexpr (kMode == kGivenScales) {
          word = code_word_any(x, __ldg(a.given_scale + e / G), live);
        } else {
          float sum = 0.f;
#pragma unroll
          for (int q = 0; q < 4; ++q)
            sum += (fabsf(x[4 * q]) + fabsf(x[4 * q + 1])) + (fabsf(x[4 * q + 2]) + fabsf(x[4 * q + 3]));
#pragma unroll
          for (int off = 1; off < kLanesPerGroup; off <<= 1) sum += __shfl_xor_sync(live, sum, off);
          s = sum * kInvG;
          const bool tiny = s < 0x1p-100f;
          word = __any_sync(live, tiny) ? (tiny ? code_word<true>(x, s) : code_word<false>(x, s))
                                        : code_word<false>(x, s);
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
        a.codes[e >> 4] = word;
        if ((lane & (kLanesPerGroup - 1)) == 0) {
          if (kMode == kAbsmean) a.scales[e / G] = s;
          a.zeros[e / G] = zc;
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty_bar(slot));
    if (++slot == kStages) {
      slot = 0;
      parity ^= 1u;
    }
  }
}

uint32_t* asched_base() {
  static std::atomic<uintptr_t> base[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  if (dev < 64) {
    const uintptr_t p = base[dev].load(std::memory_order_acquire);
    if (p != 0) return reinterpret_cast<uint32_t*>(p);
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_asched) != cudaSuccess) return nullptr;
  if (dev < 64) base[dev].store(reinterpret_cast<uintptr_t>(p), std::memory_order_release);
  return static_cast<uint32_t*>(p);
}

template <int G, int kMode>
cudaError_t launch(const AdamwArgs& a, int* status, int num_sms, cudaStream_t stream) {
  static std::atomic<uint32_t> seq{0};
  const int64_t nstages = (a.total + kStageW - 1) / kStageW;
  if (nstages <= 0) return cudaSuccess;
  if (nstages >= (int64_t{1} << 31)) return cudaErrorInvalidValue;
  const int64_t blocks = nstages < num_sms ? nstages : num_sms;
  cudaError_t e = ensure_smem_limit<adamw_requantize_kernel<G, kMode>>(kSmemBytes);
  if (e != cudaSuccess) return e;
  uint32_t* sched = asched_base();
  if (sched == nullptr) return cudaErrorInvalidSymbol;
  sched += 2 * (seq.fetch_add(1, std::memory_order_relaxed) % kSchedSlots);
  adamw_requantize_kernel<G, kMode><<<static_cast<unsigned>(blocks), kThreads, kSmemBytes, stream>>>(
      a, sched, status);
  return cudaGetLastError();
}

template <int kMode>
cudaError_t launch_mode(const AdamwArgs& a, int g, int* status, int num_sms, cudaStream_t stream) {
  switch (g) {
    case 32: return launch<32, kMode>(a, status, num_sms, stream);
    case 64: return launch<64, kMode>(a, status, num_sms, stream);
    case 128: return launch<128, kMode>(a, status, num_sms, stream);
    case 256: return launch<256, kMode>(a, status, num_sms, stream);
    case 512: return launch<512, kMode>(a, status, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_adamw_requantize(const AdamwArgs& a, int g, int* status, int num_sms,
                                    cudaStream_t stream) {
  if (a.codes == nullptr) return launch<128, kPlain>(a, status, num_sms, stream);
  return a.given_scale != nullptr ? launch_mode<kGivenScales>(a, g, status, num_sms, stream)
                                  : launch_mode<kAbsmean>(a, g, status, num_sms, stream);
}

}  // namespace tq
