// cg_internal.h -- launchers and workspace layouts shared by the library's
// translation units (host side).  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/canary_guard.h"

namespace cg {

// ---------------------------------------------------------------- device info
struct DeviceInfo {
  int device = -1;
  int sm_count = 0;
  int drift_blocks_per_sm = 0;
  int gen_blocks_per_sm = 0;
  int gen_live_blocks_per_sm = 0;
};
// Cached per current device; returns false on a CUDA error.
bool device_info(DeviceInfo *out);

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------- drift
// A work item is a chunk of at most kDriftChunk elements of one segment.
// A segment has ceil(L / kDriftChunk) items (this count sizes the
// workspace); they share the segment evenly in whole multiples of
// kDriftItemGranule elements, the bulk pipeline's stage, so that no item is
// a short remainder (L = 36,864: three items of 12,288, not 16,384 + 16,384
// + 4,096).  Only the last item of a segment may be shorter.
constexpr uint32_t kDriftChunk = 16384;
constexpr uint32_t kDriftItemGranule = 4096;
constexpr int kDriftThreads = 256;
constexpr size_t kDriftHeader = 256;   // reserved bytes at the start of the workspace

inline uint64_t drift_chunks_per_seg(uint64_t seg_len) {
  return (seg_len + kDriftChunk - 1) / kDriftChunk;
}
// Elements per item: ceil(L / items) rounded up to the granule.  It is at
// most kDriftChunk (a multiple of the granule), and items - 1 of them cover
// less than L, so the last item is never empty.
inline uint64_t drift_item_len(uint64_t seg_len) {
  const uint64_t items = drift_chunks_per_seg(seg_len);
  const uint64_t even = (seg_len + items - 1) / items;
  return (even + kDriftItemGranule - 1) / kDriftItemGranule * kDriftItemGranule;
}
inline size_t drift_ws_bytes(uint64_t n_segments, uint64_t seg_len) {
  return kDriftHeader + align_up((size_t)(n_segments * drift_chunks_per_seg(seg_len)) * 16, 256);
}


cudaError_t launch_bounded_wait_probe(uint32_t limit_us, int32_t *status, cudaStream_t stream);
bool drift_bulk_eligible(const uint16_t *acts, const float *refs, uint64_t seg_len);
// C configurations of S stages x N canaries, [C][S][N][seg_len]; scores of
// configuration c, stage s, canary n at stat * stat_stride + c N S + n S + s.
cudaError_t launch_drift_algo(const uint16_t *acts, const float *refs, uint32_t C, uint32_t S,
                              uint32_t N, uint64_t seg_len, float *scores, uint64_t stat_stride,
                              void *ws, int32_t *status, int algo, cudaStream_t stream);

// Work-item capacity of the fixed scratch array used by cg_drift_scores_noalloc.
constexpr uint64_t kNoallocDriftItems = 262144;
cudaError_t launch_drift_noalloc(const uint16_t *acts, const float *refs, uint32_t S, uint32_t N,
                                 uint64_t seg_len, float *scores, uint64_t stat_stride,
                                 cudaStream_t stream);

// ---------------------------------------------------------------- generator
constexpr uint32_t kGenStatChunk = 65536;   // elements per statistics work item
constexpr int kGenThreads = 256;
constexpr int kGenBlocksPerSm = 3;          // leaves room for a co-running drift block
constexpr uint32_t kMaxShards = 1024;
constexpr uint32_t kMaxOutliers = 256;

struct GenLayout {
  size_t outlier_mask, flip_mask, stage_sigma, seg_coef, stats, total;
  uint32_t mask_words;          // ceil(d / 32)
  uint64_t stat_chunks;         // per segment
};
GenLayout gen_layout(const cg_pipeline_desc &d);

struct GenParams {
  uint64_t seed;
  uint32_t S, N, T, d;
  uint64_t L;                   // T * d
  uint32_t config_id;
  int32_t noise, tamper;
  float sigma, lognormal, outlier_scale, tamper_param;
  uint32_t n_outlier, n_flip;   // flipped channels per malicious stage
  uint32_t mask_words;
  uint64_t stat_chunks;
  uint32_t round_keys[20];      // Philox round keys of `seed` (key + r * Weyl constants)
  int32_t recompute;            // 1: write a benign recompute of every stage into refs
  uint32_t noise_c3;            // counter word 3 of the noise stream (recompute replica)
  uint32_t mal_bits[kMaxShards / 32];
};

cudaError_t launch_generate(const GenParams &p, uint16_t *acts, float *refs, int8_t *labels,
                            void *ws, const GenLayout &lay, int32_t *status, cudaStream_t stream);

cudaError_t launch_generate_propagating(const GenParams &p, float gain, uint16_t *acts, float *refs,
                                       int8_t *labels, void *ws, const GenLayout &lay,
                                       int32_t *status, cudaStream_t stream);
cudaError_t launch_random_scores(uint64_t seed, uint32_t config_id0, uint32_t C, uint32_t N,
                                 uint32_t S, float *out, cudaStream_t stream);

cudaError_t launch_philox_words(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                                uint32_t first, uint32_t n, uint32_t *out, cudaStream_t stream);
cudaError_t launch_box_muller_pairs(const uint32_t *words, uint64_t n_pairs, float *out,
                                   cudaStream_t stream);
cudaError_t launch_philox_normals(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                                  uint32_t first, uint32_t n, float *out, cudaStream_t stream);

// ---------------------------------------------------------------- ranking
constexpr uint32_t kMaxRankShards = 1024;
cudaError_t launch_control_labels(const int8_t *labels, uint32_t C, uint32_t N, uint32_t S,
                                  uint64_t seed, uint32_t config_id0, int8_t *ctrl,
                                  int32_t *status, cudaStream_t stream);
constexpr uint32_t kMaxPooled = 16384;   // labelled scores per configuration (96 KiB of keys)
cudaError_t launch_auroc_pooled(const float *scores, const int8_t *labels, uint32_t C,
                                uint32_t N, uint32_t S, int64_t *u2, int64_t *n_mal,
                                int64_t *n_ben, double *auroc, int32_t *status,
                                cudaStream_t stream);
cudaError_t launch_auroc(const float *scores, const int8_t *labels, uint32_t C, uint32_t N,
                         uint32_t S, int64_t *u2, int64_t *gt, int64_t *eq, double *auroc,
                         int32_t *status, cudaStream_t stream);

}  // namespace cg
