// tq_api.cu — the C ABI of include/tq.h: argument checks, TMA descriptors, dispatch.
//
// Nothing here computes the method: every step runs in the kernels of
// quantize.cu, ts_gemm.cu and dw_gemm.cu. This file only validates arguments,
// encodes tensor maps for the operands, and enqueues launches on the caller's
// stream.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdarg.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <unordered_map>

#include "decode.cuh"
#include "kernels.cuh"
#include "tq.h"

namespace {

thread_local char g_err[512] = "";

tq_status fail(tq_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return st;
}

tq_status cuda_fail(cudaError_t e, const char* what) {
  return fail(TQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Per-device control words passed to every kernel (one set per device): [0] the
// status word written by kernels whose bounded waits run out, [1] test flags that
// make one role withhold one arrival (tq_test_hooks; 0 in normal use), [2..3] the
// wait limit in ns as a 64-bit value (0: the kernels' default).
__device__ __align__(16) int g_device_ctl[4];

struct DeviceInfo {
  bool ready = false;
  int num_sms = 0;
  int* status = nullptr;
};

constexpr int kMaxDevices = 64;
DeviceInfo g_devices[kMaxDevices];
std::mutex g_devices_mu;

tq_status device_info(const DeviceInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(TQ_ERR_UNSUPPORTED, "device %d", dev);
  std::lock_guard<std::mutex> lock(g_devices_mu);
  DeviceInfo& d = g_devices[dev];
  if (!d.ready) {
    int major = 0, minor = 0, sms = 0;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    if (major != 10 || minor != 3)
      return fail(TQ_ERR_UNSUPPORTED, "libtq is built for sm_103a (GB300); device %d is sm_%d%d",
                  dev, major, minor);
    void* p = nullptr;
    if ((e = cudaGetSymbolAddress(&p, g_device_ctl)) != cudaSuccess)
      return cuda_fail(e, "cudaGetSymbolAddress");
    d.num_sms = sms;
    d.status = static_cast<int*>(p);
    d.ready = true;
  }
  *out = &d;
  return TQ_OK;
}

// ---------------------------------------------------------------- tensor maps
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// 2-D row-major tensor [outer][inner] with a box of [box_outer][box_inner].
tq_status make_map(CUtensorMap* map, CUtensorMapDataType dt, int elem_bytes, const void* base,
                   int64_t inner, int64_t outer, uint32_t box_inner, uint32_t box_outer,
                   CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return fail(TQ_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner) * elem_bytes};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(TQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return TQ_OK;
}

// ---------------------------------------------------------------- checks
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int log2_group(int32_t g) {
  switch (g) {
    case 32: return 5;
    case 64: return 6;
    case 128: return 7;
    case 256: return 8;
    case 512: return 9;
    default: return -1;
  }
}

constexpr int64_t kMaxDim = (int64_t(1) << 31) - 1;  // TMA coordinates are int32

tq_status check_ptr(const void* p, const char* name) {
  if (p == nullptr) return fail(TQ_ERR_INVALID_ARG, "%s is NULL", name);
  if (!aligned16(p)) return fail(TQ_ERR_INVALID_ARG, "%s is not 16-byte aligned", name);
  return TQ_OK;
}

// dtype word: the output type in bits 0-7 (TQ_OUT_F32 / TQ_OUT_BF16), TQ_IN_F16
// for fp16 activations (x, dy) instead of bf16.
inline int out_type(int32_t dtype) { return dtype & 0xff; }
inline bool in_f16(int32_t dtype) { return (dtype & TQ_IN_F16) != 0; }
inline bool dtype_ok(int32_t dtype) {
  return (dtype & ~(0xff | TQ_IN_F16)) == 0 && (out_type(dtype) == TQ_OUT_F32 || out_type(dtype) == TQ_OUT_BF16);
}
inline CUtensorMapDataType act_map_type(int32_t dtype) {
  return in_f16(dtype) ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
}

#define TQ_TRY(expr)                 \
  do {                               \
    const tq_status st_ = (expr);    \
    if (st_ != TQ_OK) return st_;    \
  } while (0)

tq_status check_linear_shape(int64_t m, int64_t n, int64_t k, int32_t g) {
  if (m < 0 || n < 0 || k < 0)
    return fail(TQ_ERR_INVALID_ARG, "negative size (m=%lld n=%lld k=%lld)", (long long)m,
                (long long)n, (long long)k);
  if (log2_group(g) < 0) return fail(TQ_ERR_INVALID_ARG, "group size %d not in {32..512}", g);
  if (k % g != 0) return fail(TQ_ERR_INVALID_ARG, "k=%lld is not a multiple of g=%d", (long long)k, g);
  if (k % 64 != 0)
    return fail(TQ_ERR_UNSUPPORTED, "k=%lld: the linear kernels need k %% 64 == 0", (long long)k);
  if (m > kMaxDim || n > kMaxDim || k > kMaxDim)
    return fail(TQ_ERR_UNSUPPORTED, "dimension above 2^31-1");
  return TQ_OK;
}

tq_status fwd_checked(const void* x, int64_t m, int64_t k, const uint32_t* codes,
                      const float* scales, int64_t n, int32_t g, void* y, int32_t y_dtype,
                      cudaStream_t stream, const tq::TsArgs* proto) {
  if (m == 0 || n == 0) return TQ_OK;
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  const size_t ybytes = out_type(y_dtype) == TQ_OUT_BF16 ? 2 : 4;
  if (k == 0) {
    cudaError_t e = cudaMemsetAsync(y, 0, static_cast<size_t>(m) * n * ybytes, stream);
    return e == cudaSuccess ? TQ_OK : cuda_fail(e, "cudaMemsetAsync");
  }
  const int bn = tq::ts_tile_tokens(tq::kTsFwd, m);
  if (((n + 127) / 128) * ((m + bn - 1) / bn) >= (int64_t(1) << 31))
    return fail(TQ_ERR_UNSUPPORTED, "too many output tiles (m=%lld n=%lld)", (long long)m, (long long)n);
  CUtensorMap tb, tc;
  TQ_TRY(make_map(&tb, act_map_type(y_dtype), 2, x, k, m, 64, bn, CU_TENSOR_MAP_SWIZZLE_128B));
  TQ_TRY(make_map(&tc, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, codes, k / 16, n, 8, 128,
                  CU_TENSOR_MAP_SWIZZLE_NONE));
  tq::TsArgs a = *proto;
  a.codes = codes;
  a.scales = scales;
  a.out = y;
  a.status = dev->status;
  a.wn = n;
  a.wk = k;
  a.m = m;
  a.log2g = log2_group(g);
  a.out_bf16 = out_type(y_dtype) == TQ_OUT_BF16;
  a.in_f16 = in_f16(y_dtype);
  cudaError_t e = tq::launch_ts_gemm(tq::kTsFwd, bn, tb, tc, a, dev->num_sms, stream);
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "forward launch");
}

static_assert(tq::kQuantMaxMats >= TQ_MAX_BATCH, "quantize batch table");

// Tensor map of a codes matrix for the decode kernel, cached by (device, codes,
// n, k): a map encodes only the address, shape and strides, so a cached entry
// stays right for as long as the same call can be made again.
struct MapKey {
  int dev;
  const void* codes;
  int64_t n, k;
  bool operator==(const MapKey& o) const {
    return dev == o.dev && codes == o.codes && n == o.n && k == o.k;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey& x) const {
    size_t h = std::hash<const void*>()(x.codes);
    h ^= std::hash<int64_t>()(x.n) + 0x9e3779b97f4a7c15ull + (h << 6) + (h >> 2);
    h ^= std::hash<int64_t>()(x.k) + 0x9e3779b97f4a7c15ull + (h << 6) + (h >> 2);
    return h ^ static_cast<size_t>(x.dev);
  }
};

// kind 0: codes uint32 [n][k/16]; kind 1: scales fp32 [n][k/g] (k here = k/g) with
// a box of `box` groups (128 bytes: the 128-byte swizzle) x kDecodeRows rows.
tq_status decode_map(int kind, const void* base, int64_t n, int64_t k, uint32_t box,
                     CUtensorMap* out) {
  static std::mutex mu;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  const MapKey key{dev * 2 + kind, base, n, k * 1024 + box};
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      *out = it->second;
      return TQ_OK;
    }
  }
  if (kind == 0)
    TQ_TRY(make_map(out, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, base, k / 16, n,
                    tq::kDecodeSegK / 16, tq::kDecodeRows, CU_TENSOR_MAP_SWIZZLE_128B));
  else
    TQ_TRY(make_map(out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, base, k, n, box, tq::kDecodeRows,
                    CU_TENSOR_MAP_SWIZZLE_128B));
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() >= 4096) cache.clear();
  cache.emplace(key, *out);
  return TQ_OK;
}

// Forward for m <= 16 tokens: the HBM-streaming decode kernel over all matrices
// (launches of up to kDecodeMaxMats matrices each).
tq_status decode_checked(const tq_fwd_desc* descs, int32_t count, int64_t m,
                         cudaStream_t stream) {
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  thread_local tq::DecodeBatch b;
  int used = 0, used_smaps = 0;
  // one activation type per call (checked by the callers)
  b.in_f16 = count > 0 && in_f16(descs[0].y_dtype);
  auto flush = [&]() -> tq_status {
    if (used == 0) return TQ_OK;
    b.status = dev->status;
    b.count = used;
    b.m = static_cast<int32_t>(m);
    b.total_units = 0;
    used = 0;
    used_smaps = 0;
    cudaError_t e = tq::launch_decode(b, dev->num_sms, stream);
    return e == cudaSuccess ? TQ_OK : cuda_fail(e, "decode launch");
  };
  for (int32_t i = 0; i < count; ++i) {
    const tq_fwd_desc& d = descs[i];
    if (d.n == 0) continue;
    if (d.k == 0) {
      const size_t yb = out_type(d.y_dtype) == TQ_OUT_BF16 ? 2 : 4;
      cudaError_t e = cudaMemsetAsync(d.y, 0, static_cast<size_t>(m) * d.n * yb, stream);
      if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
      continue;
    }
    if (d.n >= (int64_t(1) << 31)) return fail(TQ_ERR_UNSUPPORTED, "too many decode rows");
    if (d.k > (int64_t(1) << 30)) return fail(TQ_ERR_UNSUPPORTED, "decode reduction longer than 2^30");
    const int log2g = log2_group(d.g);
    const int64_t gpr = d.k >> log2g;
    const int mode = gpr % 4 != 0                 ? tq::kDecodeScale4
                     : gpr <= tq::kDecodeWinGroups ? tq::kDecodeScaleUnit
                                                   : tq::kDecodeScaleWin;
    // code maps from the bottom of maps[], window-mode scale maps from the top
    const int nmaps = mode == tq::kDecodeScaleWin ? 2 : 1;
    if (used + used_smaps + nmaps > tq::kDecodeMaxMats) TQ_TRY(flush());
    TQ_TRY(decode_map(0, d.codes, d.n, d.k, 0, &b.maps[used]));
    tq::DecodeMat& dm = b.mats[used++];
    dm.scales = d.scales;
    dm.x = d.x;
    dm.y = d.y;
    dm.n = d.n;
    dm.k = d.k;
    dm.log2g = log2g;
    dm.y_bf16 = out_type(d.y_dtype) == TQ_OUT_BF16;
    dm.unit0 = 0;
    dm.scale_mode = static_cast<int16_t>(mode);
    dm.smap = 0;
    if (mode == tq::kDecodeScaleWin) {
      // rows of k/g floats (a multiple of 16 bytes), scales 16-byte aligned (checked)
      dm.smap = tq::kDecodeMaxMats - 1 - used_smaps++;
      TQ_TRY(decode_map(1, d.scales, d.n, gpr, tq::kDecodeWinGroups, &b.maps[dm.smap]));
    }
  }
  return flush();
}

tq_status check_fwd_args(const void* x, int64_t m, int64_t k, const uint32_t* codes,
                         const float* scales, int64_t n, int32_t g, const void* y,
                         int32_t y_dtype) {
  TQ_TRY(check_linear_shape(m, n, k, g));
  if (!dtype_ok(y_dtype)) return fail(TQ_ERR_INVALID_ARG, "y_dtype %d", y_dtype);
  if (m == 0 || n == 0) return TQ_OK;
  TQ_TRY(check_ptr(y, "y"));
  if (k == 0) return TQ_OK;
  TQ_TRY(check_ptr(x, "x"));
  TQ_TRY(check_ptr(codes, "codes"));
  TQ_TRY(check_ptr(scales, "scales"));
  return TQ_OK;
}

}  // namespace

namespace tq {
// dw_gemm.cu: zero the stream-K completion counters (after a launch gave up on a
// wait, when the CTA that would have reset them may not have run). Synchronous.
cudaError_t reset_dw_counters();
}  // namespace tq

extern "C" {

TQ_API const char* tq_last_error(void) { return g_err; }

TQ_API const char* tq_version(void) { return "tq 0.1 (sm_103a)"; }

tq_status check_quantize_args(const float* w, int64_t n, int64_t k, int32_t g, const uint32_t* codes,
                               const float* scales, const int32_t* zero_counts) {
  if (n < 0 || k < 0) return fail(TQ_ERR_INVALID_ARG, "negative size");
  if (log2_group(g) < 0) return fail(TQ_ERR_INVALID_ARG, "group size %d not in {32..512}", g);
  if (k % 16 != 0) return fail(TQ_ERR_INVALID_ARG, "k=%lld is not a multiple of 16", (long long)k);
  if (k % g != 0) return fail(TQ_ERR_INVALID_ARG, "k=%lld is not a multiple of g=%d", (long long)k, g);
  if (n == 0 || k == 0) return TQ_OK;
  if (n > INT64_MAX / k) return fail(TQ_ERR_INVALID_ARG, "n*k overflows");
  TQ_TRY(check_ptr(w, "w"));
  TQ_TRY(check_ptr(codes, "codes"));
  TQ_TRY(check_ptr(scales, "scales"));
  TQ_TRY(check_ptr(zero_counts, "zero_counts"));
  return TQ_OK;
}

TQ_API tq_status tq_quantize(const float* w, int64_t n, int64_t k, int32_t g, uint32_t* codes,
                             float* scales, int32_t* zero_counts, void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_quantize_args(w, n, k, g, codes, scales, zero_counts));
  if (n == 0 || k == 0) return TQ_OK;
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_quantize(w, n, k, g, codes, scales, zero_counts, dev->status,
                                      dev->num_sms, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "quantize launch");
}

TQ_API tq_status tq_quantize_with_transpose(const float* w, int64_t n, int64_t k, int32_t g,
                                            uint32_t* codes, float* scales, int32_t* zero_counts,
                                            uint32_t* codes_t, void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_quantize_args(w, n, k, g, codes, scales, zero_counts));
  if (n == 0 || k == 0) return TQ_OK;
  if (n > kMaxDim || k > kMaxDim) return fail(TQ_ERR_UNSUPPORTED, "dimension too large");
  TQ_TRY(check_ptr(codes_t, "codes_t"));
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_quantize_t(w, n, k, g, codes, scales, zero_counts, codes_t,
                                        dev->status, dev->num_sms,
                                        static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "quantize + transpose launch");
}

TQ_API tq_status tq_quantize_decoupled(const float* w, int64_t n, int64_t k, int32_t g,
                                       const float* row_factor, uint32_t* codes, float* scales,
                                       int32_t* zero_counts, void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_quantize_args(w, n, k, g, codes, scales, zero_counts));
  if (n == 0 || k == 0) return TQ_OK;
  if (row_factor != nullptr && (reinterpret_cast<uintptr_t>(row_factor) & 3) != 0)
    return fail(TQ_ERR_INVALID_ARG, "row_factor is not 4-byte aligned");
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_quantize(w, n, k, g, codes, scales, zero_counts, dev->status,
                                      dev->num_sms, static_cast<cudaStream_t>(stream), row_factor);
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "quantize launch");
}

TQ_API tq_status tq_alpha_grad(const float* dw, const uint32_t* codes, int64_t n, int64_t k,
                               int32_t g, float* dalpha, void* stream) {
  g_err[0] = 0;
  if (n < 0 || k < 0) return fail(TQ_ERR_INVALID_ARG, "negative size");
  if (log2_group(g) < 0) return fail(TQ_ERR_INVALID_ARG, "group size %d not in {32..512}", g);
  if (k % g != 0) return fail(TQ_ERR_INVALID_ARG, "k=%lld is not a multiple of g=%d", (long long)k, g);
  if (n == 0 || k == 0) return TQ_OK;
  if (n > INT64_MAX / k) return fail(TQ_ERR_INVALID_ARG, "n*k overflows");
  TQ_TRY(check_ptr(dw, "dw"));
  TQ_TRY(check_ptr(codes, "codes"));
  if (dalpha == nullptr || (reinterpret_cast<uintptr_t>(dalpha) & 3) != 0)
    return fail(TQ_ERR_INVALID_ARG, "dalpha is NULL or not 4-byte aligned");
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_alpha_grad(dw, codes, n, k, g, dalpha, dev->num_sms,
                                        static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "alpha_grad launch");
}

TQ_API tq_status tq_quantize_with_scales(const float* w, int64_t n, int64_t k, int32_t g,
                                         const float* scales, uint32_t* codes,
                                         int32_t* zero_counts, void* stream) {
  g_err[0] = 0;
  // the scales are an input here; the absmean check of tq_quantize covers the rest
  TQ_TRY(check_quantize_args(w, n, k, g, codes, scales, zero_counts));
  if (n == 0 || k == 0) return TQ_OK;
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_quantize(w, n, k, g, codes, nullptr, zero_counts, dev->status,
                                      dev->num_sms, static_cast<cudaStream_t>(stream), nullptr,
                                      scales);
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "quantize launch");
}

TQ_API tq_status tq_scale_grad(const float* w, const float* dw, const uint32_t* codes,
                               const float* scales, int64_t n, int64_t k, int32_t g,
                               float* dscales, void* stream) {
  g_err[0] = 0;
  if (n < 0 || k < 0) return fail(TQ_ERR_INVALID_ARG, "negative size");
  if (log2_group(g) < 0) return fail(TQ_ERR_INVALID_ARG, "group size %d not in {32..512}", g);
  if (k % g != 0) return fail(TQ_ERR_INVALID_ARG, "k=%lld is not a multiple of g=%d", (long long)k, g);
  if (n == 0 || k == 0) return TQ_OK;
  if (n > INT64_MAX / k) return fail(TQ_ERR_INVALID_ARG, "n*k overflows");
  TQ_TRY(check_ptr(w, "w"));
  TQ_TRY(check_ptr(dw, "dw"));
  TQ_TRY(check_ptr(codes, "codes"));
  if (scales == nullptr || (reinterpret_cast<uintptr_t>(scales) & 3) != 0)
    return fail(TQ_ERR_INVALID_ARG, "scales is NULL or not 4-byte aligned");
  if (dscales == nullptr || (reinterpret_cast<uintptr_t>(dscales) & 3) != 0)
    return fail(TQ_ERR_INVALID_ARG, "dscales is NULL or not 4-byte aligned");
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_scale_grad(w, dw, codes, scales, n, k, g, dscales, dev->num_sms,
                                        static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "scale_grad launch");
}

TQ_API tq_status tq_quantize_batched(const tq_quant_desc* descs, int32_t count, int32_t g,
                                     void* stream) {
  g_err[0] = 0;
  if (count < 0 || count > TQ_MAX_BATCH)
    return fail(TQ_ERR_INVALID_ARG, "count %d not in [0, %d]", count, TQ_MAX_BATCH);
  if (count > 0 && descs == nullptr) return fail(TQ_ERR_INVALID_ARG, "descs is NULL");
  if (log2_group(g) < 0) return fail(TQ_ERR_INVALID_ARG, "group size %d not in {32..512}", g);
  thread_local tq::QuantBatch<tq::kQuantMaxMats> b;
  b.count = 0;
  for (int32_t i = 0; i < count; ++i) {
    const tq_quant_desc& d = descs[i];
    const tq_status st = check_quantize_args(d.w, d.n, d.k, g, d.codes, d.scales, d.zero_counts);
    if (st != TQ_OK) {
      char msg[sizeof(g_err)];
      snprintf(msg, sizeof(msg), "%s", g_err);
      return fail(st, "descs[%d]: %s", i, msg);
    }
    if (d.n == 0 || d.k == 0) continue;
    b.mats[b.count++] = tq::QuantMat{d.w, d.codes, d.scales, d.zero_counts, d.n * d.k, 0, nullptr, d.k};
  }
  if (b.count == 0) return TQ_OK;
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_quantize_batched(b, g, dev->status, dev->num_sms,
                                              static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "quantize launch");
}

namespace {
// AdamW hyperparameters checked and turned into the kernel's fp32 step constants
// (computed in fp64, rounded once).
tq_status adamw_const(const tq_adamw_hparams* hp, tq::AdamwConst* c) {
  if (hp == nullptr) return fail(TQ_ERR_INVALID_ARG, "hparams is NULL");
  if (hp->step < 1) return fail(TQ_ERR_INVALID_ARG, "step %lld < 1", (long long)hp->step);
  const double lr = hp->lr, b1 = hp->beta1, b2 = hp->beta2, eps = hp->eps;
  const double wd = hp->weight_decay, gs = hp->grad_scale;
  if (!(lr >= 0 && lr < 1e30) || !(b1 >= 0 && b1 < 1) || !(b2 >= 0 && b2 < 1) ||
      !(eps > 0 && eps < 1e30) || !(wd >= 0 && wd < 1e30) || !(gs >= 0 && gs < 1e30))
    return fail(TQ_ERR_INVALID_ARG, "hyperparameters out of range");
  const double t = static_cast<double>(hp->step);
  c->b1 = static_cast<float>(b1);
  c->omb1 = static_cast<float>(1.0 - b1);
  c->b2 = static_cast<float>(b2);
  c->omb2 = static_cast<float>(1.0 - b2);
  c->decay = static_cast<float>(1.0 - lr * wd);
  c->step_size = static_cast<float>(lr / (1.0 - pow(b1, t)));
  c->inv_bc2_sqrt = static_cast<float>(1.0 / sqrt(1.0 - pow(b2, t)));
  c->eps = static_cast<float>(eps);
  c->grad_scale = static_cast<float>(gs);
  return TQ_OK;
}

tq_status adamw_launch(tq::AdamwArgs& a, int32_t g, void* stream) {
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_adamw_requantize(a, g, dev->status, dev->num_sms,
                                              static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "adamw launch");
}
}  // namespace

TQ_API tq_status tq_adamw_requantize(float* w, const float* grad, float* m, float* v, int64_t n,
                                     int64_t k, int32_t g, const tq_adamw_hparams* hp,
                                     uint32_t* codes, float* scales, int32_t* zero_counts,
                                     void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_quantize_args(w, n, k, g, codes, scales, zero_counts));
  tq::AdamwArgs a{};
  TQ_TRY(adamw_const(hp, &a.c));
  if (n == 0 || k == 0) return TQ_OK;
  TQ_TRY(check_ptr(grad, "grad"));
  TQ_TRY(check_ptr(m, "m"));
  TQ_TRY(check_ptr(v, "v"));
  a.w = w;
  a.grad = grad;
  a.m = m;
  a.v = v;
  a.codes = codes;
  a.scales = scales;
  a.zeros = zero_counts;
  a.total = n * k;
  return adamw_launch(a, g, stream);
}

TQ_API tq_status tq_adamw_requantize_with_scales(float* w, const float* grad, float* m, float* v,
                                                 int64_t n, int64_t k, int32_t g,
                                                 const tq_adamw_hparams* hp, const float* scales,
                                                 uint32_t* codes, int32_t* zero_counts,
                                                 void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_quantize_args(w, n, k, g, codes, scales, zero_counts));
  tq::AdamwArgs a{};
  TQ_TRY(adamw_const(hp, &a.c));
  if (n == 0 || k == 0) return TQ_OK;
  TQ_TRY(check_ptr(grad, "grad"));
  TQ_TRY(check_ptr(m, "m"));
  TQ_TRY(check_ptr(v, "v"));
  a.w = w;
  a.grad = grad;
  a.m = m;
  a.v = v;
  a.codes = codes;
  a.zeros = zero_counts;
  a.given_scale = scales;
  a.total = n * k;
  return adamw_launch(a, g, stream);
}

TQ_API tq_status tq_adamw(float* p, const float* grad, float* m, float* v, int64_t count,
                          const tq_adamw_hparams* hp, void* stream) {
  g_err[0] = 0;
  if (count < 0) return fail(TQ_ERR_INVALID_ARG, "negative count");
  if (count % 16 != 0) return fail(TQ_ERR_INVALID_ARG, "count=%lld is not a multiple of 16", (long long)count);
  tq::AdamwArgs a{};
  TQ_TRY(adamw_const(hp, &a.c));
  if (count == 0) return TQ_OK;
  TQ_TRY(check_ptr(p, "p"));
  TQ_TRY(check_ptr(grad, "grad"));
  TQ_TRY(check_ptr(m, "m"));
  TQ_TRY(check_ptr(v, "v"));
  a.w = p;
  a.grad = grad;
  a.m = m;
  a.v = v;
  a.total = count;  // codes == nullptr: no requantization
  return adamw_launch(a, 128, stream);
}

TQ_API tq_status tq_linear_fwd(const void* x, int64_t m, int64_t k, const uint32_t* codes,
                               const float* scales, int64_t n, int32_t g, void* y,
                               int32_t y_dtype, void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_fwd_args(x, m, k, codes, scales, n, g, y, y_dtype));
  if (m >= 1 && m <= 16 && n > 0) {
    tq_fwd_desc d{x, codes, scales, y, n, k, g, y_dtype};
    return decode_checked(&d, 1, m, static_cast<cudaStream_t>(stream));
  }
  tq::TsArgs proto{};
  return fwd_checked(x, m, k, codes, scales, n, g, y, y_dtype, static_cast<cudaStream_t>(stream),
                     &proto);
}

TQ_API tq_status tq_linear_fwd_batched(const tq_fwd_desc* descs, int32_t count, int64_t m,
                                       void* stream) {
  g_err[0] = 0;
  if (count < 0 || count > TQ_MAX_BATCH)
    return fail(TQ_ERR_INVALID_ARG, "count %d not in [0, %d]", count, TQ_MAX_BATCH);
  if (count == 0) return TQ_OK;
  if (descs == nullptr) return fail(TQ_ERR_INVALID_ARG, "descs is NULL");
  if (m < 1 || m > 16) return fail(TQ_ERR_INVALID_ARG, "batched decode needs 1 <= m <= 16");
  for (int32_t i = 0; i < count; ++i) {
    const tq_fwd_desc& d = descs[i];
    const tq_status st = check_fwd_args(d.x, m, d.k, d.codes, d.scales, d.n, d.g, d.y, d.y_dtype);
    if (st != TQ_OK) {
      char msg[512];
      snprintf(msg, sizeof(msg), "descs[%d]: %s", i, g_err);
      return fail(st, "%s", msg);
    }
    if (in_f16(d.y_dtype) != in_f16(descs[0].y_dtype))
      return fail(TQ_ERR_INVALID_ARG, "descs[%d]: activation type differs from descs[0]", i);
  }
  return decode_checked(descs, count, m, static_cast<cudaStream_t>(stream));
}

TQ_API tq_status tq_codes_transpose(const uint32_t* codes, int64_t n, int64_t k,
                                    uint32_t* codes_t, void* stream) {
  g_err[0] = 0;
  if (n < 0 || k < 0) return fail(TQ_ERR_INVALID_ARG, "negative size");
  if (k % 16 != 0) return fail(TQ_ERR_INVALID_ARG, "k=%lld is not a multiple of 16", (long long)k);
  if (n == 0 || k == 0) return TQ_OK;
  if (n > kMaxDim || k > kMaxDim || (n + 127) / 128 > 65535)
    return fail(TQ_ERR_UNSUPPORTED, "dimension too large");
  TQ_TRY(check_ptr(codes, "codes"));
  TQ_TRY(check_ptr(codes_t, "codes_t"));
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = tq::launch_transpose_codes(codes, n, k, codes_t, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? TQ_OK : cuda_fail(e, "transpose launch");
}

// Arguments of the backward, checked before anything is enqueued.
tq_status check_bwd_args(const void* dy, const void* x, int64_t m, int64_t n, int64_t k,
                         const uint32_t* codes, const uint32_t* codes_t, const float* scales,
                         int32_t g, const void* dx, int32_t dx_dtype, const float* dw) {
  TQ_TRY(check_linear_shape(m, n, k, g));
  if (n % 8 != 0)
    return fail(TQ_ERR_UNSUPPORTED, "n=%lld: the backward kernels need n %% 8 == 0", (long long)n);
  if (!dtype_ok(dx_dtype)) return fail(TQ_ERR_INVALID_ARG, "dx_dtype %d", dx_dtype);
  if (dx == nullptr && dw == nullptr) return fail(TQ_ERR_INVALID_ARG, "dx and dw are both NULL");
  const bool want_dx = dx != nullptr && m > 0 && k > 0;
  const bool want_dw = dw != nullptr && n > 0 && k > 0;
  if (want_dx) {
    TQ_TRY(check_ptr(dx, "dx"));
    if (n > 0) {
      TQ_TRY(check_ptr(dy, "dy"));
      if (codes_t == nullptr) TQ_TRY(check_ptr(codes, "codes"));
      else TQ_TRY(check_ptr(codes_t, "codes_t"));
      TQ_TRY(check_ptr(scales, "scales"));
    }
  }
  if (want_dw) {
    TQ_TRY(check_ptr(dw, "dw"));
    if (m > 0) {
      TQ_TRY(check_ptr(dy, "dy"));
      TQ_TRY(check_ptr(x, "x"));
    }
  }
  return TQ_OK;
}

TQ_API tq_status tq_linear_bwd(const void* dy, const void* x, int64_t m, int64_t n, int64_t k,
                               const uint32_t* codes, const uint32_t* codes_t,
                               const float* scales, int32_t g, void* dx, int32_t dx_dtype,
                               float* dw, int32_t accumulate_dw, void* stream) {
  g_err[0] = 0;
  TQ_TRY(check_bwd_args(dy, x, m, n, k, codes, codes_t, scales, g, dx, dx_dtype, dw));
  const bool want_dx = dx != nullptr && m > 0 && k > 0;
  const bool want_dw = dw != nullptr && n > 0 && k > 0;
  if (!want_dx && !want_dw) return TQ_OK;
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  if (want_dx) {
    const size_t dxb = out_type(dx_dtype) == TQ_OUT_BF16 ? 2 : 4;
    if (n == 0) {
      cudaError_t e = cudaMemsetAsync(dx, 0, static_cast<size_t>(m) * k * dxb, st);
      if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    } else {
      const int bn = tq::ts_tile_tokens(tq::kTsDx, m);
      if (((k + 127) / 128) * ((m + bn - 1) / bn) >= (int64_t(1) << 31))
        return fail(TQ_ERR_UNSUPPORTED, "too many output tiles (m=%lld k=%lld)", (long long)m, (long long)k);
      CUtensorMap tb, tc;
      TQ_TRY(make_map(&tb, act_map_type(dx_dtype), 2, dy, n, m, 64, bn,
                      CU_TENSOR_MAP_SWIZZLE_128B));
      const int64_t ldt = 4 * ((n + 63) / 64);  // codes_t row length (words)
      if (codes_t != nullptr)
        TQ_TRY(make_map(&tc, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, codes_t, ldt, k, 8, 128,
                        CU_TENSOR_MAP_SWIZZLE_NONE));
      else
        TQ_TRY(make_map(&tc, CU_TENSOR_MAP_DATA_TYPE_UINT32, 4, codes, k / 16, n, 8, 128,
                        CU_TENSOR_MAP_SWIZZLE_NONE));
      tq::TsArgs a{};
      a.codes = codes_t != nullptr ? codes_t : codes;
      a.scales = scales;
      a.out = dx;
      a.status = dev->status;
      a.wn = n;
      a.wk = k;
      a.m = m;
      a.log2g = log2_group(g);
      a.out_bf16 = out_type(dx_dtype) == TQ_OUT_BF16;
      a.in_f16 = in_f16(dx_dtype);
      cudaError_t e = tq::launch_ts_gemm(codes_t != nullptr ? tq::kTsDxT : tq::kTsDx, bn, tb, tc,
                                         a, dev->num_sms, st);
      if (e != cudaSuccess) return cuda_fail(e, "dX launch");
    }
  }
  if (want_dw) {
    if (m == 0) {
      if (!accumulate_dw) {
        cudaError_t e = cudaMemsetAsync(dw, 0, static_cast<size_t>(n) * k * 4, st);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
      }
    } else {
      if (((n + tq::kDwTileN - 1) / tq::kDwTileN) * ((k + tq::kDwTileK - 1) / tq::kDwTileK) >=
          (int64_t(1) << 31))
        return fail(TQ_ERR_UNSUPPORTED, "too many dW tiles (n=%lld k=%lld)", (long long)n, (long long)k);
      CUtensorMap tx, tdy;
      TQ_TRY(make_map(&tx, act_map_type(dx_dtype), 2, x, k, m, 64, 64,
                      CU_TENSOR_MAP_SWIZZLE_128B));
      TQ_TRY(make_map(&tdy, act_map_type(dx_dtype), 2, dy, n, m, 64, 64,
                      CU_TENSOR_MAP_SWIZZLE_128B));
      tq::DwArgs a{};
      a.dw = dw;
      a.status = dev->status;
      a.m = m;
      a.n = n;
      a.k = k;
      a.accumulate = accumulate_dw != 0;
      a.in_f16 = in_f16(dx_dtype);
      cudaError_t e = tq::launch_dw_gemm(tx, tdy, a, dev->num_sms, st);
      if (e != cudaSuccess) return cuda_fail(e, "dW launch");
    }
  }
  return TQ_OK;
}

TQ_API tq_status tq_device_status(void* stream) {
  g_err[0] = 0;
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int v = 0;
  if ((e = cudaMemcpy(&v, dev->status, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "status read");
  if (v != 0) {
    // Work of every stream of the device ends before the reset: a dW launch still
    // running on another stream would otherwise race with it.
    if ((e = cudaDeviceSynchronize()) != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
    const int zero = 0;
    if ((e = cudaMemcpy(dev->status, &zero, sizeof(int), cudaMemcpyHostToDevice)) != cudaSuccess)
      return cuda_fail(e, "status clear");
    // a dW launch that gave up may have left tile counters of its stream-K tail set
    if ((e = tq::reset_dw_counters()) != cudaSuccess) return cuda_fail(e, "dW counter reset");
    return fail(TQ_ERR_TIMEOUT, "a kernel wait ran out (device status %d)", v);
  }
  return TQ_OK;
}

TQ_API tq_status tq_test_hooks(int64_t wait_limit_ns, uint32_t flags) {
  g_err[0] = 0;
  if (wait_limit_ns < 0) return fail(TQ_ERR_INVALID_ARG, "negative wait limit");
  if ((flags & ~7u) != 0) return fail(TQ_ERR_INVALID_ARG, "unknown test flags 0x%x", flags);
  const DeviceInfo* dev = nullptr;
  TQ_TRY(device_info(&dev));
  cudaError_t e = cudaDeviceSynchronize();  // no kernel may be reading the words
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  int words[3];
  words[0] = static_cast<int>(flags);
  const uint64_t lim = static_cast<uint64_t>(wait_limit_ns);
  memcpy(&words[1], &lim, sizeof(lim));
  if ((e = cudaMemcpy(dev->status + 1, words, sizeof(words), cudaMemcpyHostToDevice)) != cudaSuccess)
    return cuda_fail(e, "test hooks write");
  return TQ_OK;
}

}  // extern "C"

// ---------------------------------------------------------------- no-alloc backward
// Scratch for the transposed codes of tq_linear_bwd_noalloc: a file-scope device
// array, so the caller allocates nothing. One per device; calls that use it must
// not overlap in time on one device (keep them on one stream).
constexpr int64_t kNoAllocWords = int64_t(4) << 20;  // 16 MB of uint32 words
static __device__ __align__(256) uint32_t g_codes_t_scratch[kNoAllocWords];

namespace {
tq_status noalloc_scratch(uint32_t** out) {
  static std::atomic<uintptr_t> base[kMaxDevices];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(TQ_ERR_UNSUPPORTED, "device %d", dev);
  uintptr_t p = base[dev].load(std::memory_order_acquire);
  if (p == 0) {
    void* a = nullptr;
    if ((e = cudaGetSymbolAddress(&a, g_codes_t_scratch)) != cudaSuccess)
      return cuda_fail(e, "cudaGetSymbolAddress");
    p = reinterpret_cast<uintptr_t>(a);
    base[dev].store(p, std::memory_order_release);
  }
  *out = reinterpret_cast<uint32_t*>(p);
  return TQ_OK;
}
}  // namespace

TQ_API tq_status tq_linear_bwd_noalloc(const void* dy, const void* x, int64_t m, int64_t n,
                                       int64_t k, const uint32_t* codes, const float* scales,
                                       int32_t g, void* dx, int32_t dx_dtype, float* dw,
                                       int32_t accumulate_dw, void* stream) {
  g_err[0] = 0;
  const bool want_dx = dx != nullptr && m > 0 && k > 0 && n > 0;
  if (!want_dx)  // nothing to transpose: exactly tq_linear_bwd
    return tq_linear_bwd(dy, x, m, n, k, codes, nullptr, scales, g, dx, dx_dtype, dw,
                         accumulate_dw, stream);
  TQ_TRY(check_bwd_args(dy, x, m, n, k, codes, nullptr, scales, g, dx, dx_dtype, dw));
  const int64_t ldt = 4 * ((n + 63) / 64);
  if (k > kNoAllocWords / ldt)
    return fail(TQ_ERR_UNSUPPORTED,
                "transposed codes of n=%lld k=%lld need %lld words, scratch holds %lld; pass "
                "codes_t to tq_linear_bwd instead",
                (long long)n, (long long)k, (long long)(ldt * k), (long long)kNoAllocWords);
  // the device and architecture check before the scratch's address is looked up
  // (an unsupported device gets TQ_ERR_UNSUPPORTED, as from every entry point)
  const DeviceInfo* devinfo = nullptr;
  TQ_TRY(device_info(&devinfo));
  uint32_t* scratch = nullptr;
  TQ_TRY(noalloc_scratch(&scratch));
  const cudaError_t e =
      tq::launch_transpose_codes(codes, n, k, scratch, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "transpose launch");
  return tq_linear_bwd(dy, x, m, n, k, codes, scratch, scales, g, dx, dx_dtype, dw,
                       accumulate_dw, stream);
}
