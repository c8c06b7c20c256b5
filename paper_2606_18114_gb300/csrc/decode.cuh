// decode.cuh — the decode kernel's batch descriptor and launcher (internal to
// libtq): the forward for m <= 16 tokens over one or many matrices in one launch.
// Apart from kernels.cuh so that the other kernels' sources do not change with it.
#pragma once

#include "kernels.cuh"

namespace tq {

struct DecodeMat {
  const float* scales;    // fp32 [n][k/g]
  const void* x;          // bf16 [m][k]
  void* y;                // [m][n], fp32 or bf16
  int64_t n, k;           // k % 64 == 0
  int32_t log2g;
  int32_t unit0;          // first unit of this matrix in the batch (set by the launcher)
  int16_t y_bf16;
  int16_t scale_mode;     // how the kernel fetches scales (host-set, kDecodeScale*)
  int32_t smap;           // window mode: index of the scales' tensor map in maps[]
};

// Scale fetch modes: per segment in 4-byte pieces (k/g % 4 != 0); per window of
// kDecodeWinGroups groups of all the unit's rows, one 2-D TMA box (k/g % 4 == 0,
// k/g > kDecodeWinGroups); a whole unit in one bulk copy (k/g % 4 == 0,
// k/g <= kDecodeWinGroups).
constexpr int kDecodeScale4 = 0, kDecodeScaleWin = 1, kDecodeScaleUnit = 2;
constexpr int kDecodeMaxMats = 128;  // tensor maps per launch (they travel as parameters)
constexpr int kDecodeRows = 256;    // weight rows per work unit
constexpr int kDecodeSegK = 512;    // k per streamed segment (128-byte code rows)
constexpr int kDecodeWinGroups = 32;  // groups per row of a scale window (128 bytes)

struct DecodeBatch {
  // maps[d], d < count: codes of matrix d as uint32 [n][k/16], box {kDecodeSegK / 16
  // words, kDecodeRows rows}, 128-byte swizzle. From the top down (maps[smap]): the
  // scales of the window-mode matrices as fp32 [n][k/g], box {kDecodeWinGroups,
  // kDecodeRows}, 128-byte swizzle. count + (window-mode matrices) <= kDecodeMaxMats.
  CUtensorMap maps[kDecodeMaxMats];
  DecodeMat mats[kDecodeMaxMats];
  int* status;            // device status word (timeouts)
  int32_t count;
  int32_t m;              // tokens, 1..16
  int32_t total_units;    // sum over matrices of ceil(n / kDecodeRows) (set by the launcher)
  int32_t slot_bytes;     // shared-memory ring slot: codes, scales, x (set by the launcher)
  int32_t scale_bytes;    // scale area of a slot
  int32_t stages;         // ring slots
  int32_t ubuf_bytes;     // one unit- or window-scale buffer (two are kept)
  int32_t in_f16;         // 1: fp16 activations in every matrix (else bf16)
  // pieces of k per block of rows (set by the launcher): 1, a persistent grid
  // claiming units; P > 1, clusters of P CTAs, CTA p of a cluster taking piece p
  // of one block's segments, the first CTA adding the others' partial sums
  int32_t pieces;
};

// Reorders b.mats / b.maps (decreasing k) and sets unit0 and total_units.
cudaError_t launch_decode(DecodeBatch& batch, int num_sms, cudaStream_t stream);

}  // namespace tq
