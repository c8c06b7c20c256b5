// kernels.cuh — launchers of the sm_103a kernels (internal to libtq).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace tq {

// Raise a kernel's dynamic shared-memory limit once per device (the attribute
// persists; setting it on every launch costs host time on the launch path).
template <auto kKernel>
cudaError_t ensure_smem_limit(int bytes) {
  static std::atomic<uint64_t> done{0};  // bit d: set on device d (d < 64), per kernel
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t{1} << dev) : 0;
  if (bit != 0 && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kKernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && bit != 0) done.fetch_or(bit, std::memory_order_release);
  return e;
}

// quantize.cu ----------------------------------------------------------------
// row_factor (fp32 [n] or null): the codes of row r are decided against the
// threshold row_factor[r] * s instead of s (the decoupled quantizer); scales stay s.
// given_scale (fp32 [n][k/g] or null): the codes are decided against these scales
// (the learnable-scale variant) and scales is not written.
cudaError_t launch_quantize(const float* w, int64_t n, int64_t k, int g, uint32_t* codes,
                            float* scales, int32_t* zeros, int* status, int num_sms,
                            cudaStream_t stream, const float* row_factor = nullptr,
                            const float* given_scale = nullptr);

// Many matrices (same group size) in one launch.
struct QuantMat {
  const float* w;   // fp32 [n][k], flat
  uint32_t* codes;  // uint32 [n][k/16]
  float* scales;    // fp32 [n][k/g]
  int32_t* zeros;   // int32 [n][k/g]
  int64_t total;    // n * k
  int64_t stage0;   // first stage of this matrix (set by the launcher)
  const float* row_factor;  // null, or fp32 [n]: per-row threshold factor
  int64_t k;        // row length (for row_factor)
  const float* given_scale;  // null, or fp32 [n][k/g]: decide against these scales
                             // (scales is then not written)
};

// dalpha[n][k/g] = sum over each group of dw * code (the decoupled quantizer's
// magnitude gradient).
cudaError_t launch_alpha_grad(const float* dw, const uint32_t* codes, int64_t n, int64_t k, int g,
                              float* dalpha, int num_sms, cudaStream_t stream);

// dscale[n][k/g] = sum over each group of dw * (c - q [|w| < |s|]), q = w / s: the
// gradient of a learnable scale through W^ = s * round(clip(w / s)) with the
// rounding passed straight through.
cudaError_t launch_scale_grad(const float* w, const float* dw, const uint32_t* codes,
                              const float* scales, int64_t n, int64_t k, int g, float* dscale,
                              int num_sms, cudaStream_t stream);

template <int kMax>
struct QuantBatch {
  QuantMat mats[kMax];
  int64_t nstages;  // set by the launcher
  int32_t count;
  int32_t pad;
};

constexpr int kQuantMaxMats = 256;

cudaError_t launch_quantize_batched(QuantBatch<kQuantMaxMats>& batch, int g, int* status,
                                    int num_sms, cudaStream_t stream);

// launch_quantize followed, in the same cooperative launch, by launch_transpose_codes
// of the codes it wrote.
cudaError_t launch_quantize_t(const float* w, int64_t n, int64_t k, int g, uint32_t* codes,
                              float* scales, int32_t* zeros, uint32_t* codes_t, int* status,
                              int num_sms, cudaStream_t stream);

// codes [n][k/16] -> codes_t [k][4 * ceil(n / 64)] (the codes of W^T).
cudaError_t launch_transpose_codes(const uint32_t* codes, int64_t n, int64_t k, uint32_t* codes_t,
                                   cudaStream_t stream);

// adamw.cu -------------------------------------------------------------------
// Fused AdamW step + requantize of one weight matrix (flat, n * k weights).
struct AdamwConst {     // fp32 step constants (computed in fp64 on the host)
  float b1, omb1;       // beta1, 1 - beta1
  float b2, omb2;       // beta2, 1 - beta2
  float decay;          // 1 - lr * weight_decay
  float step_size;      // lr / (1 - beta1^t)
  float inv_bc2_sqrt;   // 1 / sqrt(1 - beta2^t)
  float eps;
  float grad_scale;     // multiplies the gradient (gradient clipping)
};

struct AdamwArgs {
  float* w;             // fp32 [n][k], updated in place
  const float* grad;    // fp32 [n][k]
  float* m;             // fp32 [n][k], updated in place
  float* v;             // fp32 [n][k], updated in place
  uint32_t* codes;      // uint32 [n][k/16] of the new w; null: no requantization
  float* scales;        // fp32 [n][k/g]
  int32_t* zeros;       // int32 [n][k/g]
  int64_t total;        // n * k
  AdamwConst c;
  const float* given_scale;  // null, or fp32 [n][k/g]: requantize against these
};

cudaError_t launch_adamw_requantize(const AdamwArgs& a, int g, int* status, int num_sms,
                                    cudaStream_t stream);

// ts_gemm.cu -----------------------------------------------------------------
// Ternary x bf16 products with the expanded ternary weights as the tensor-memory
// A operand. kTsFwd: out[m][n] = sum_k x[m][k] w^[n][k] (B = x, rows = n).
// kTsDx: out[m][k] = sum_n dy[m][n] w^[n][k] (B = dy, rows = k), codes read as is.
// kTsDxT: the same product with the transposed codes (codes_t) as input.
enum TsMode : int { kTsFwd = 0, kTsDx = 1, kTsDxT = 2 };

struct TsArgs {
  const uint32_t* codes;  // uint32 [wn][wk/16] (fwd, dx) or codes_t [wk][ldt] (dxt)
  const float* scales;    // fp32 [wn][wk/g]
  void* out;              // [m][rows], fp32 or bf16
  int* status;            // device status word (timeouts)
  int64_t wn, wk;         // shape of the latent weight matrix W [wn][wk]
  int64_t m;              // tokens
  int32_t log2g;          // log2 of the group size
  int32_t out_bf16;       // 1: bf16 output
  int32_t in_f16;         // 1: fp16 activations (else bf16)
};

// Tile of the activation operand along the token dimension.
int ts_tile_tokens(int mode, int64_t m);

// tmap_b: bf16 activations [m][red] with box {64, bn}, 128-byte swizzle.
// tmap_codes: uint32 codes [wn][wk/16] with box {8, 128} (8 words x 128 rows).
// Persistent: min(tiles, num_sms) CTAs.
cudaError_t launch_ts_gemm(int mode, int bn, const CUtensorMap& tmap_b,
                           const CUtensorMap& tmap_codes, const TsArgs& args, int num_sms,
                           cudaStream_t stream);

// decode.cu: declared in decode.cuh.

// dw_gemm.cu -----------------------------------------------------------------
// dW[n][k] (+)= sum_m dy[m][n] x[m][k], both operands MN-major from TMA.
struct DwArgs {
  float* dw;       // fp32 [n][k]
  int* status;
  int64_t m, n, k;
  int32_t accumulate;
  int32_t in_f16;  // 1: fp16 dy and x (else bf16)
};

constexpr int kDwTileK = 128;  // lanes: input features (one CTA of a pair)
constexpr int kDwPairK = 2 * kDwTileK;  // input features of a CTA pair's tile
constexpr int kDwTileN = 256;  // columns: output features
constexpr int kDwMaxCtas = 160;  // grid cap (stream-K workspace: two half-tiles per CTA)
size_t dw_smem_bytes();

// tmap_x: bf16 x [m][k] box {64, 64}; tmap_dy: bf16 dy [m][n] box {64, 64};
// both with the 128-byte swizzle. Persistent: clusters of two CTAs (one pair per
// two SMs), min(tiles, resident pairs) pairs.
cudaError_t launch_dw_gemm(const CUtensorMap& tmap_x, const CUtensorMap& tmap_dy,
                           const DwArgs& args, int num_sms, cudaStream_t stream);

}  // namespace tq
