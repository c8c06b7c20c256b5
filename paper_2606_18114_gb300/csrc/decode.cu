// decode.cu — W1.58A16 forward for few tokens (m <= 16): an HBM-streaming kernel
// over the packed codes of one or many matrices in one launch (§8: at small batch
// the layer is bound by weight traffic; 2-bit codes + fp32 group scales are 0.28
// bytes per weight at g = 128).
//
// Work unit = 16 consecutive weight rows of one matrix over its whole K. Each CTA
// owns a contiguous range of units, balanced by their number of 128-wide chunks
// of K (host-computed), so an SM works through one or two matrices at a time and
// their x stays in L1. Warps take units from the range with a shared-memory
// counter. A warp streams its units as a flat sequence of chunks: the codes of a
// chunk (16 rows x 32 bytes) are one 16-byte cp.async per lane, zero-filled past
// the matrix, into a per-warp ring of kDepth chunks (~128 KB per SM in flight
// without holding registers); a per-warp queue hands the units claimed by the
// prefetch cursor to the consuming cursor.
//
// Per chunk a warp runs eight mma.sync.m16n8k16 (bf16 in, fp32 accumulate) with
// the expanded weights as the 16 x 16 A operand and up to 8 tokens as the n8 B
// operand (two B tiles for 9..16 tokens), in two independent accumulator chains.
// The reduction index of the MMA is permuted identically on both operands so that
// lane (g, t) (g = lane / 4, t = lane % 4) consumes exactly code words 2t, 2t+1 of
// the chunk for rows g and g + 8 — reduction offsets 32t .. 32t + 31 — and the
// contiguous 64 bytes x[token g][32t .. 32t + 31]: MMA kb takes offsets
// 32t + 4kb + {0,1} for fragment slots (2t, 2t+1) and 32t + 4kb + {2,3} for slots
// (2t+8, 2t+9).
//
// Expansion: pair j of a code word -> bf16x2 (2c, 2c) by ((w << (14 - 2j)) &
// 0xC000C000) (layout of include/tq.h). For g >= 128 a chunk lies in one group and
// the partial sums of a group are scaled by s/2 in fp32 (exact scale); for g <= 64
// the groups of a chunk meet inside one MMA, so the expansion multiplies by
// bf16(s)/2 as the prefill kernels do.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace tq {
namespace {

constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kDepth = 16;                 // chunks in flight per warp
constexpr int kChunkBytes = 16 * 32;       // 16 rows x 8 code words
constexpr int kQueue = kDepth + 1;         // units claimed ahead of the consumer
constexpr int kSmemBytes = kWarps * kDepth * kChunkBytes;

__device__ __forceinline__ uint32_t bmul2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Pair j of a code word as a bf16x2 of (2c, 2c): the mask keeps the pair's two
// fields, the multiplication by mul = 2^(14 - 2j) moves them to bits 14-15 and
// 30-31 (exact, the fields are 16 bits apart). mul is a register whose value the
// compiler does not see, so the move runs as an integer multiply on the FMA pipe
// instead of a shift on the ALU pipe, which the mask already loads.
__device__ __forceinline__ uint32_t pair_bits(uint32_t w, int j, uint32_t mul) {
  return (w & (0x00030003u << (2 * j))) * mul;
}

__device__ __forceinline__ uint32_t opaque(uint32_t v) {
  uint32_t r;
  asm volatile("mov.b32 %0, %1;" : "=r"(r) : "r"(v));
  return r;
}

__device__ __forceinline__ void mma16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 16-byte global -> shared copy; bytes beyond src_bytes (0 or 16) are zero-filled.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ uint32_t half_scale_bf16x2(float s) {
  const __nv_bfloat16 h = __float2bfloat16_rn(0.5f * s);
  const uint32_t u = __bfloat16_as_ushort(h);
  return u | (u << 16);
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

template <bool kTwoTiles>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ DecodeBatch b) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ int next_unit;
  __shared__ int queue[kWarps][kQueue];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) &
                                             ~static_cast<uintptr_t>(127));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int m = b.m;
  const int uend = b.cta_unit[blockIdx.x + 1];
  if (threadIdx.x == 0) next_unit = b.cta_unit[blockIdx.x];
  __syncthreads();
  uint8_t* ring = smem + warp * kDepth * kChunkBytes;
  const uint32_t ring_u32 = static_cast<uint32_t>(__cvta_generic_to_shared(ring));
  int* q = queue[warp];
  uint32_t mul[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) mul[j] = opaque(1u << (14 - 2 * j));

  // ------------------------------------------------------------ prefetch cursor
  // Lane l copies 16 bytes per chunk: row l / 2 of the unit, words 4 (l & 1) .. + 3.
  const int crow = lane >> 1, chalf = lane & 1;
  int qtail = 0;            // units claimed (queue writes)
  int pu = -1;              // unit being prefetched (-1: stream exhausted)
  int pc = 0, pnc = 0;      // its next chunk / chunk count
  const uint32_t* psrc = nullptr;
  bool prow = false;        // this lane's row exists
  bool phalf = false;       // this lane's half of the last chunk lies past k
  auto claim = [&]() {
    int u = 0;
    if (lane == 0) u = atomicAdd(&next_unit, 1);
    u = __shfl_sync(0xffffffffu, u, 0);
    if (u >= uend) {
      pu = -1;
      return;
    }
    const int d = find_mat(b, u);
    const DecodeMat& mat = b.mats[d];
    const int64_t row = static_cast<int64_t>(u - mat.unit0) * 16 + crow;
    pu = u;
    pc = 0;
    pnc = static_cast<int>((mat.k + 127) >> 7);
    prow = row < mat.n;
    phalf = chalf && (mat.k & 127);
    psrc = mat.codes + (prow ? row : 0) * (mat.k >> 4) + chalf * 4;
    if (lane == 0) q[qtail % kQueue] = u;
    ++qtail;
  };
  auto issue = [&](int slot) {
    if (pu >= 0) {
      const bool in = prow && !(phalf && pc + 1 == pnc);
      cp_async16(ring_u32 + slot * kChunkBytes + crow * 32 + chalf * 16, psrc + 8 * pc,
                 in ? 16u : 0u);
      if (++pc == pnc) claim();
    }
    cp_async_commit();  // one group per slot, empty past the end of the stream
  };

  claim();
  for (int s = 0; s < kDepth - 1; ++s) issue(s);

  // ------------------------------------------------------------ consumer
  int qhead = 0;
  int slot = 0;
  while (qhead < qtail) {
    __syncwarp();
    const int u = q[qhead % kQueue];
    ++qhead;
    const int d = find_mat(b, u);
    const DecodeMat& mat = b.mats[d];
    const int64_t n = mat.n, k = mat.k;
    const int64_t r0 = static_cast<int64_t>(u - mat.unit0) * 16;
    const int64_t ra = r0 + g, rb = r0 + g + 8;
    const bool va = ra < n, vb = rb < n;
    const int log2g = mat.log2g;
    const int64_t gpr = k >> log2g;
    const float* sa = mat.scales + (va ? ra : 0) * gpr;
    const float* sb = mat.scales + (vb ? rb : 0) * gpr;
    const bool ta = g < m, tb = kTwoTiles && (g + 8 < m);
    const uint4* xa = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(mat.x) +
                                                     static_cast<int64_t>(ta ? g : 0) * k + 32 * t);
    const uint4* xb = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(mat.x) +
                                                     static_cast<int64_t>(tb ? g + 8 : 0) * k + 32 * t);
    const int nc = static_cast<int>((k + 127) >> 7);
    // a lane's 32 offsets of the last chunk lie past k when k % 128 == 64 and t >= 2
    const bool tail_lane = (k & 127) && t >= 2;
    float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
    float p0[4] = {0.f, 0.f, 0.f, 0.f}, p1[4] = {0.f, 0.f, 0.f, 0.f};
    float q0[4] = {0.f, 0.f, 0.f, 0.f}, q1[4] = {0.f, 0.f, 0.f, 0.f};

    if (log2g >= 7) {
      // exact path: one scale per row per group of (g / 128) chunks
      const int cpg = 1 << (log2g - 7);
      int left = cpg;
      int gi = 0;
      for (int c = 0; c < nc; ++c) {
        issue((slot + kDepth - 1) % kDepth);
        cp_async_wait<kDepth - 1>();
        __syncwarp();
        const uint8_t* st = ring + slot * kChunkBytes;
        const uint2 wa = *reinterpret_cast<const uint2*>(st + g * 32 + 8 * t);
        const uint2 wb = *reinterpret_cast<const uint2*>(st + (g + 8) * 32 + 8 * t);
        uint4 xv[4], yv[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          xv[i] = ta ? __ldg(xa + 16 * c + i) : make_uint4(0, 0, 0, 0);
          if (kTwoTiles) yv[i] = tb ? __ldg(xb + 16 * c + i) : make_uint4(0, 0, 0, 0);
        }
        const uint32_t* xr = reinterpret_cast<const uint32_t*>(xv);
        const uint32_t* yr = reinterpret_cast<const uint32_t*>(yv);
#pragma unroll
        for (int kb = 0; kb < 8; ++kb) {
          const uint32_t ua = kb < 4 ? wa.x : wa.y, ub = kb < 4 ? wb.x : wb.y;
          const int j = 2 * (kb & 3);
          const uint32_t a0 = pair_bits(ua, j, mul[j]), a1 = pair_bits(ub, j, mul[j]);
          const uint32_t a2 = pair_bits(ua, j + 1, mul[j + 1]), a3 = pair_bits(ub, j + 1, mul[j + 1]);
          if (kb & 1) {
            mma16816(q0, a0, a1, a2, a3, xr[2 * kb], xr[2 * kb + 1]);
            if (kTwoTiles) mma16816(q1, a0, a1, a2, a3, yr[2 * kb], yr[2 * kb + 1]);
          } else {
            mma16816(p0, a0, a1, a2, a3, xr[2 * kb], xr[2 * kb + 1]);
            if (kTwoTiles) mma16816(p1, a0, a1, a2, a3, yr[2 * kb], yr[2 * kb + 1]);
          }
        }
        __syncwarp();
        slot = slot + 1 == kDepth ? 0 : slot + 1;
        if (--left == 0) {
          // group closed: acc += (s / 2) * partial; rows g (slots 0, 1), g + 8 (2, 3)
          left = cpg;
          const float ha = va ? 0.5f * __ldg(sa + gi) : 0.f;
          const float hb = vb ? 0.5f * __ldg(sb + gi) : 0.f;
          ++gi;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float h = i < 2 ? ha : hb;
            acc0[i] = fmaf(h, p0[i] + q0[i], acc0[i]);
            p0[i] = q0[i] = 0.f;
            if (kTwoTiles) {
              acc1[i] = fmaf(h, p1[i] + q1[i], acc1[i]);
              p1[i] = q1[i] = 0.f;
            }
          }
        }
      }
    } else {
      // g = 32 or 64: lane t's offsets 32t .. 32t + 31 of a chunk lie in one group
      const int gshift = 7 - log2g;  // groups per chunk = 1 << gshift
      for (int c = 0; c < nc; ++c) {
        issue((slot + kDepth - 1) % kDepth);
        cp_async_wait<kDepth - 1>();
        __syncwarp();
        const bool kin = !(tail_lane && c + 1 == nc);
        const uint8_t* st = ring + slot * kChunkBytes;
        const uint2 wa = *reinterpret_cast<const uint2*>(st + g * 32 + 8 * t);
        const uint2 wb = *reinterpret_cast<const uint2*>(st + (g + 8) * 32 + 8 * t);
        const int64_t gi = (static_cast<int64_t>(c) << gshift) + (t >> (log2g - 5));
        const uint32_t ha = (va && kin) ? half_scale_bf16x2(__ldg(sa + gi)) : 0u;
        const uint32_t hb = (vb && kin) ? half_scale_bf16x2(__ldg(sb + gi)) : 0u;
        uint4 xv[4], yv[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          xv[i] = (ta && kin) ? __ldg(xa + 16 * c + i) : make_uint4(0, 0, 0, 0);
          if (kTwoTiles) yv[i] = (tb && kin) ? __ldg(xb + 16 * c + i) : make_uint4(0, 0, 0, 0);
        }
        const uint32_t* xr = reinterpret_cast<const uint32_t*>(xv);
        const uint32_t* yr = reinterpret_cast<const uint32_t*>(yv);
#pragma unroll
        for (int kb = 0; kb < 8; ++kb) {
          const uint32_t ua = kb < 4 ? wa.x : wa.y, ub = kb < 4 ? wb.x : wb.y;
          const int j = 2 * (kb & 3);
          const uint32_t a0 = bmul2(pair_bits(ua, j, mul[j]), ha), a1 = bmul2(pair_bits(ub, j, mul[j]), hb);
          const uint32_t a2 = bmul2(pair_bits(ua, j + 1, mul[j + 1]), ha), a3 = bmul2(pair_bits(ub, j + 1, mul[j + 1]), hb);
          if (kb & 1) {
            mma16816(q0, a0, a1, a2, a3, xr[2 * kb], xr[2 * kb + 1]);
            if (kTwoTiles) mma16816(q1, a0, a1, a2, a3, yr[2 * kb], yr[2 * kb + 1]);
          } else {
            mma16816(acc0, a0, a1, a2, a3, xr[2 * kb], xr[2 * kb + 1]);
            if (kTwoTiles) mma16816(acc1, a0, a1, a2, a3, yr[2 * kb], yr[2 * kb + 1]);
          }
        }
        __syncwarp();
        slot = slot + 1 == kDepth ? 0 : slot + 1;
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc0[i] += q0[i];
        if (kTwoTiles) acc1[i] += q1[i];
      }
    }

    // C fragment: rows g (slots 0, 1) and g + 8 (slots 2, 3), tokens 2t and 2t + 1
    auto store = [&](int token, int64_t row, float v) {
      if (token < m && row < n) {
        if (mat.y_bf16)
          static_cast<__nv_bfloat16*>(mat.y)[token * n + row] = __float2bfloat16_rn(v);
        else
          static_cast<float*>(mat.y)[token * n + row] = v;
      }
    };
    store(2 * t, ra, acc0[0]);
    store(2 * t + 1, ra, acc0[1]);
    store(2 * t, rb, acc0[2]);
    store(2 * t + 1, rb, acc0[3]);
    if (kTwoTiles) {
      store(8 + 2 * t, ra, acc1[0]);
      store(8 + 2 * t + 1, ra, acc1[1]);
      store(8 + 2 * t, rb, acc1[2]);
      store(8 + 2 * t + 1, rb, acc1[3]);
    }
  }
  cp_async_wait<0>();  // nothing may still write this warp's ring when it exits
}

}  // namespace

cudaError_t launch_decode(DecodeBatch& b, int num_sms, cudaStream_t stream) {
  if (b.total_units <= 0) return cudaSuccess;
  int64_t blocks = (static_cast<int64_t>(b.total_units) + kWarps - 1) / kWarps;
  if (blocks > num_sms) blocks = num_sms;
  if (blocks > kDecodeMaxCtas) blocks = kDecodeMaxCtas;
  // Split the units into `blocks` contiguous ranges of about equal chunk count.
  int64_t work = 0;
  for (int d = 0; d < b.count; ++d) {
    const int64_t units = (b.mats[d].n + 15) / 16;
    work += units * ((b.mats[d].k + 127) / 128);
  }
  int c = 0;
  int64_t acc = 0;
  b.cta_unit[0] = 0;
  for (int d = 0; d < b.count && c + 1 < blocks; ++d) {
    const int64_t units = (b.mats[d].n + 15) / 16;
    const int64_t per = (b.mats[d].k + 127) / 128;
    for (int64_t u = 0; u < units && c + 1 < blocks; ++u) {
      acc += per;
      // close range c once it holds its share (c + 1) * work / blocks
      while (c + 1 < blocks && acc * blocks >= (c + 1) * work) {
        b.cta_unit[++c] = b.mats[d].unit0 + static_cast<int32_t>(u) + 1;
      }
    }
  }
  while (c < blocks) b.cta_unit[++c] = b.total_units;
  const size_t smem = kSmemBytes + 128;
  cudaError_t e;
  if (b.m > 8) {
    e = ensure_smem_limit<decode_kernel<true>>(static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    decode_kernel<true><<<static_cast<unsigned>(blocks), kThreads, smem, stream>>>(b);
  } else {
    e = ensure_smem_limit<decode_kernel<false>>(static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    decode_kernel<false><<<static_cast<unsigned>(blocks), kThreads, smem, stream>>>(b);
  }
  return cudaGetLastError();
}

}  // namespace tq
