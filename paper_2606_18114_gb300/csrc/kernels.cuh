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
cudaError_t launch_quantize(const float* w, int64_t n, int64_t k, int g, uint32_t* codes,
                            float* scales, int32_t* zeros, int* status, int num_sms,
                            cudaStream_t stream);

// Many matrices (same group size) in one launch.
struct QuantMat {
  const float* w;   // fp32 [n][k], flat
  uint32_t* codes;  // uint32 [n][k/16]
  float* scales;    // fp32 [n][k/g]
  int32_t* zeros;   // int32 [n][k/g]
  int64_t total;    // n * k
  int64_t stage0;   // first stage of this matrix (set by the launcher)
};

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

// codes [n][k/16] -> codes_t [k][4 * ceil(n / 64)] (the codes of W^T).
cudaError_t launch_transpose_codes(const uint32_t* codes, int64_t n, int64_t k, uint32_t* codes_t,
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
};

// Tile of the activation operand along the token dimension.
int ts_tile_tokens(int mode, int64_t m);

// tmap_b: bf16 activations [m][red] with box {64, bn}, 128-byte swizzle.
// tmap_codes: uint32 codes [wn][wk/16] with box {8, 128} (8 words x 128 rows).
// Persistent: min(tiles, num_sms) CTAs.
cudaError_t launch_ts_gemm(int mode, int bn, const CUtensorMap& tmap_b,
                           const CUtensorMap& tmap_codes, const TsArgs& args, int num_sms,
                           cudaStream_t stream);

// decode.cu ------------------------------------------------------------------
// Forward for m <= 16 tokens over one or many matrices in one launch.
struct DecodeMat {
  const uint32_t* codes;  // uint32 [n][k/16]
  const float* scales;    // fp32 [n][k/g]
  const void* x;          // bf16 [m][k]
  void* y;                // [m][n], fp32 or bf16
  int64_t n, k;           // k % 64 == 0
  int32_t log2g;
  int32_t y_bf16;
  int32_t unit0;          // first 16-row unit of this matrix in the batch
  int32_t pad;
};

constexpr int kDecodeMaxMats = 256;
constexpr int kDecodeMaxCtas = 256;

struct DecodeBatch {
  DecodeMat mats[kDecodeMaxMats];
  int32_t cta_unit[kDecodeMaxCtas + 1];  // CTA c owns units [cta_unit[c], cta_unit[c + 1])
  int* status;            // device status word (timeouts)
  int32_t count;
  int32_t m;              // tokens, 1..16
  int32_t total_units;    // sum over matrices of ceil(n / 16)
  int32_t pad;
};

cudaError_t launch_decode(DecodeBatch& batch, int num_sms, cudaStream_t stream);

// dw_gemm.cu -----------------------------------------------------------------
// dW[n][k] (+)= sum_m dy[m][n] x[m][k], both operands MN-major from TMA.
struct DwArgs {
  float* dw;       // fp32 [n][k]
  int* status;
  int64_t m, n, k;
  int32_t accumulate;
};

constexpr int kDwTileK = 128;  // lanes: input features
constexpr int kDwTileN = 256;  // columns: output features
size_t dw_smem_bytes();

// tmap_x: bf16 x [m][k] box {64, 64}; tmap_dy: bf16 dy [m][n] box {64, 64};
// both with the 128-byte swizzle. Persistent: min(tiles, num_sms) CTAs.
cudaError_t launch_dw_gemm(const CUtensorMap& tmap_x, const CUtensorMap& tmap_dy,
                           const DwArgs& args, int num_sms, cudaStream_t stream);

}  // namespace tq
