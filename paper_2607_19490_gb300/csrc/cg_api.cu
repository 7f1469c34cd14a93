// cg_api.cu -- the C ABI declared in include/canary_guard.h: argument
// validation on the host, workspace sizing and kernel dispatch.  No entry
// point allocates device memory or synchronises (except cg_read_status).
#include <math.h>
#include <mutex>
#include <string.h>

#include "cg_internal.h"

#include <nvtx3/nvToolsExt.h>

// An NVTX range around every public call (visible in Nsight timelines; a
// no-op unless a tool is attached).
namespace {
struct NvtxRange {
  explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};
}  // namespace
#define CG_TRACE(name) NvtxRange cg_nvtx_range_(name)

static_assert(CG_NOALLOC_MAX_WORK_ITEMS == cg::kNoallocDriftItems,
              "public limit and scratch size disagree");
static_assert(CG_NOALLOC_CHUNK_ELEMENTS == cg::kDriftChunk, "public chunk and kernel chunk disagree");

namespace cg {

int drift_occupancy();
int gen_occupancy();
int gen_live_occupancy();

bool device_info(DeviceInfo *out) {
  static std::mutex mu;
  static DeviceInfo cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return false;
  std::lock_guard<std::mutex> lock(mu);
  if (dev < 64 && cache[dev].device == dev) {
    *out = cache[dev];
    return true;
  }
  DeviceInfo info;
  info.device = dev;
  if (cudaDeviceGetAttribute(&info.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return false;
  info.drift_blocks_per_sm = drift_occupancy();
  info.gen_blocks_per_sm = gen_occupancy();
  info.gen_live_blocks_per_sm = gen_live_occupancy();
  if (info.drift_blocks_per_sm < 1 || info.gen_blocks_per_sm < 1 || info.gen_live_blocks_per_sm < 1)
    return false;
  if (dev < 64) cache[dev] = info;
  *out = info;
  return true;
}

}  // namespace cg

namespace {

inline bool aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

inline cg_status from_cuda(cudaError_t e) { return e == cudaSuccess ? CG_OK : CG_ERR_CUDA; }

// true for memory allocated on a device (cudaMalloc and friends)
bool is_device_memory(const void *p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice;
}

cg_status check_desc(const cg_pipeline_desc *d) {
  if (!d) return CG_ERR_INVALID_ARG;
  if (d->n_shards < 1 || d->hidden < 1 || d->n_canaries < 1 || d->tokens < 1)
    return CG_ERR_INVALID_ARG;
  if (d->n_shards > cg::kMaxShards) return CG_ERR_UNSUPPORTED;
  const uint64_t L = (uint64_t)d->tokens * d->hidden;
  if (L >= (1ull << 34)) return CG_ERR_UNSUPPORTED;
  if ((uint64_t)d->n_shards * d->n_canaries >= (1ull << 32)) return CG_ERR_UNSUPPORTED;
  if (d->config_id >= (1u << 30)) return CG_ERR_INVALID_ARG;
  if (d->n_malicious >= d->n_shards) return CG_ERR_INVALID_ARG;
  if (d->n_malicious > 0 && !d->malicious) return CG_ERR_INVALID_ARG;
  if (d->noise != CG_NOISE_MULT && d->noise != CG_NOISE_PAPER) return CG_ERR_INVALID_ARG;
  if (d->tamper < CG_TAMPER_ADDITIVE || d->tamper > CG_TAMPER_SCALE) return CG_ERR_INVALID_ARG;
  if (d->n_outlier > d->hidden) return CG_ERR_INVALID_ARG;
  if (d->n_outlier > cg::kMaxOutliers) return CG_ERR_UNSUPPORTED;
  if (!isfinite(d->benign_sigma) || d->benign_sigma < 0.f) return CG_ERR_INVALID_ARG;
  if (!isfinite(d->shard_sigma_lognormal) || d->shard_sigma_lognormal < 0.f)
    return CG_ERR_INVALID_ARG;
  if (!isfinite(d->outlier_scale) || !isfinite(d->tamper_param)) return CG_ERR_INVALID_ARG;
  if (d->tamper == CG_TAMPER_SIGNFLIP_CHANNELS &&
      !(d->tamper_param > 0.f && d->tamper_param <= 1.f))
    return CG_ERR_INVALID_ARG;
  for (uint32_t i = 0; i < d->n_malicious; ++i) {
    const int32_t s = d->malicious[i];
    if (s < 0 || (uint32_t)s >= d->n_shards) return CG_ERR_INVALID_ARG;
    for (uint32_t j = 0; j < i; ++j)
      if (d->malicious[j] == s) return CG_ERR_INVALID_ARG;
  }
  return CG_OK;
}

cg::GenParams make_params(const cg_pipeline_desc &d, const cg::GenLayout &lay) {
  cg::GenParams p;
  memset(&p, 0, sizeof(p));
  p.seed = d.seed;
  p.S = d.n_shards;
  p.N = d.n_canaries;
  p.T = d.tokens;
  p.d = d.hidden;
  p.L = (uint64_t)d.tokens * d.hidden;
  p.config_id = d.config_id;
  p.noise = d.noise;
  p.tamper = d.tamper;
  p.sigma = d.benign_sigma;
  p.lognormal = d.shard_sigma_lognormal;
  p.outlier_scale = d.outlier_scale;
  p.tamper_param = d.tamper_param;
  p.n_outlier = d.n_outlier;
  // max(1, round-half-up(p d)) flipped channels, evaluated in double
  double r = floor((double)d.tamper_param * (double)d.hidden + 0.5);
  uint32_t nf = r < 1.0 ? 1u : (r > (double)d.hidden ? d.hidden : (uint32_t)r);
  p.n_flip = nf;
  p.mask_words = lay.mask_words;
  p.stat_chunks = lay.stat_chunks;
  {
    uint32_t k0 = (uint32_t)d.seed, k1 = (uint32_t)(d.seed >> 32);
    for (int r = 0; r < 10; ++r) {   // Philox round keys (SC'11 key schedule)
      p.round_keys[2 * r] = k0;
      p.round_keys[2 * r + 1] = k1;
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
  }
  for (uint32_t i = 0; i < d.n_malicious; ++i) {
    const uint32_t s = (uint32_t)d.malicious[i];
    p.mal_bits[s >> 5] |= 1u << (s & 31);
  }
  return p;
}

// Argument checks and kernel choice shared by the drift entry points: C
// configurations of S stages x N canaries, [C][S][N][seg_len].
cg_status drift_scores_checked(const uint16_t *d_acts, const float *d_refs, uint32_t n_configs,
                               uint32_t n_shards, uint32_t n_canaries, uint64_t seg_len,
                               float *d_scores, uint64_t stat_stride, void *d_ws, size_t ws_bytes,
                               int32_t *d_status, int32_t algo, cg_stream_t stream) {
  if (!d_acts || !d_refs || !d_scores || n_configs == 0 || n_shards == 0 || n_canaries == 0 ||
      seg_len == 0)
    return CG_ERR_INVALID_ARG;
  if (algo < CG_DRIFT_AUTO || algo > CG_DRIFT_BULK_2CTA) return CG_ERR_INVALID_ARG;
  const uint64_t n_seg = (uint64_t)n_configs * n_shards * n_canaries;
  if (seg_len > (1ull << 40) || n_seg > (1ull << 31)) return CG_ERR_UNSUPPORTED;
  if (stat_stride < n_seg) return CG_ERR_INVALID_ARG;
  if (!aligned(d_acts, 16) || !aligned(d_refs, 16) || !aligned(d_scores, 4) ||
      (d_status && !aligned(d_status, 4)))
    return CG_ERR_ALIGNMENT;
  if (!d_ws || ws_bytes < cg::drift_ws_bytes(n_seg, seg_len)) return CG_ERR_WORKSPACE;
  if (!aligned(d_ws, 16)) return CG_ERR_ALIGNMENT;
  // The bulk-copy pipelines take device memory only (8-element aligned
  // segments); anything else streams through registers.
  const bool bulk_ok = cg::drift_bulk_eligible(d_acts, d_refs, seg_len) &&
                       is_device_memory(d_acts) && is_device_memory(d_refs);
  if ((algo == CG_DRIFT_BULK || algo == CG_DRIFT_BULK_2CTA) && !bulk_ok)
    return CG_ERR_UNSUPPORTED;
  if (algo == CG_DRIFT_AUTO) algo = bulk_ok ? CG_DRIFT_BULK : CG_DRIFT_STREAM;
  return from_cuda(cg::launch_drift_algo(d_acts, d_refs, n_configs, n_shards, n_canaries,
                                         seg_len, d_scores, stat_stride, d_ws, d_status, algo,
                                         (cudaStream_t)stream));
}

}  // namespace

extern "C" {

const char *cg_status_string(cg_status s) {
  switch (s) {
    case CG_OK: return "CG_OK";
    case CG_ERR_INVALID_ARG: return "CG_ERR_INVALID_ARG: invalid argument";
    case CG_ERR_ALIGNMENT: return "CG_ERR_ALIGNMENT: device pointer misaligned";
    case CG_ERR_WORKSPACE: return "CG_ERR_WORKSPACE: workspace missing or too small";
    case CG_ERR_NAN_SCORE: return "CG_ERR_NAN_SCORE: a labelled score is NaN";
    case CG_ERR_CUDA: return "CG_ERR_CUDA: CUDA launch or runtime error";
    case CG_ERR_TIMEOUT: return "CG_ERR_TIMEOUT: a bounded device wait gave up";
    case CG_ERR_UNSUPPORTED: return "CG_ERR_UNSUPPORTED: size beyond this build's limits";
    case CG_ERR_NO_BENIGN: return "CG_ERR_NO_BENIGN: a control canary had no benign stage";
  }
  return "unknown cg_status";
}

int cg_abi_version(void) { return 1; }

cg_status cg_philox_words(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                          uint32_t first_block, uint32_t n_blocks, uint32_t *d_out,
                          cg_stream_t stream) {
  CG_TRACE("cg_philox_words");
  if (!d_out || n_blocks == 0) return CG_ERR_INVALID_ARG;
  if (!aligned(d_out, 16)) return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_philox_words(seed, c1, c2, c3, first_block, n_blocks, d_out,
                                           (cudaStream_t)stream));
}

cg_status cg_philox_normals(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                            uint32_t first_block, uint32_t n_blocks, float *d_out,
                            cg_stream_t stream) {
  CG_TRACE("cg_philox_normals");
  if (!d_out || n_blocks == 0) return CG_ERR_INVALID_ARG;
  if (!aligned(d_out, 16)) return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_philox_normals(seed, c1, c2, c3, first_block, n_blocks, d_out,
                                             (cudaStream_t)stream));
}

cg_status cg_box_muller_pairs(const uint32_t *d_words, uint64_t n_pairs, float *d_out,
                              cg_stream_t stream) {
  CG_TRACE("cg_box_muller_pairs");
  if (!d_words || !d_out || n_pairs == 0) return CG_ERR_INVALID_ARG;
  if (!aligned(d_words, 8) || !aligned(d_out, 8)) return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_box_muller_pairs(d_words, n_pairs, d_out, (cudaStream_t)stream));
}

cg_status cg_generate_workspace_size(const cg_pipeline_desc *desc, size_t *bytes) {
  if (!bytes) return CG_ERR_INVALID_ARG;
  cg_status st = check_desc(desc);
  if (st != CG_OK) return st;
  *bytes = cg::gen_layout(*desc).total;
  return CG_OK;
}

cg_status cg_generate_pipeline(const cg_pipeline_desc *desc, uint16_t *d_acts, float *d_refs,
                               int8_t *d_labels, void *d_ws, size_t ws_bytes, int32_t *d_status,
                               cg_stream_t stream) {
  CG_TRACE("cg_generate_pipeline");
  cg_status st = check_desc(desc);
  if (st != CG_OK) return st;
  if (!d_acts || !d_refs) return CG_ERR_INVALID_ARG;
  if (!aligned(d_acts, 16) || !aligned(d_refs, 16) || (d_status && !aligned(d_status, 4)))
    return CG_ERR_ALIGNMENT;
  const cg::GenLayout lay = cg::gen_layout(*desc);
  if (!d_ws || ws_bytes < lay.total) return CG_ERR_WORKSPACE;
  if (!aligned(d_ws, 16)) return CG_ERR_ALIGNMENT;

  cg::GenParams p = make_params(*desc, lay);
  return from_cuda(cg::launch_generate(p, d_acts, d_refs, d_labels, d_ws, lay, d_status,
                                       (cudaStream_t)stream));
}

cg_status cg_generate_recompute(const cg_pipeline_desc *desc, uint32_t replica, float *d_out,
                                void *d_ws, size_t ws_bytes, int32_t *d_status,
                                cg_stream_t stream) {
  CG_TRACE("cg_generate_recompute");
  cg_status st = check_desc(desc);
  if (st != CG_OK) return st;
  if (!d_out) return CG_ERR_INVALID_ARG;
  if (!aligned(d_out, 16) || (d_status && !aligned(d_status, 4))) return CG_ERR_ALIGNMENT;
  const cg::GenLayout lay = cg::gen_layout(*desc);
  if (!d_ws || ws_bytes < lay.total) return CG_ERR_WORKSPACE;
  if (!aligned(d_ws, 16)) return CG_ERR_ALIGNMENT;
  cg::GenParams p = make_params(*desc, lay);
  memset(p.mal_bits, 0, sizeof(p.mal_bits));   // the recompute is honest on every stage
  p.recompute = 1;
  p.noise_c3 = replica;
  return from_cuda(cg::launch_generate(p, nullptr, d_out, nullptr, d_ws, lay, d_status,
                                       (cudaStream_t)stream));
}

cg_status cg_generate_propagating(const cg_pipeline_desc *desc, float gain, uint16_t *d_acts,
                                  float *d_refs, int8_t *d_labels, void *d_ws, size_t ws_bytes,
                                  int32_t *d_status, cg_stream_t stream) {
  CG_TRACE("cg_generate_propagating");
  cg_status st = check_desc(desc);
  if (st != CG_OK) return st;
  if (!isfinite(gain)) return CG_ERR_INVALID_ARG;
  if (!d_acts || !d_refs) return CG_ERR_INVALID_ARG;
  if (!aligned(d_acts, 16) || !aligned(d_refs, 16) || (d_status && !aligned(d_status, 4)))
    return CG_ERR_ALIGNMENT;
  const cg::GenLayout lay = cg::gen_layout(*desc);
  if (!d_ws || ws_bytes < lay.total) return CG_ERR_WORKSPACE;
  if (!aligned(d_ws, 16)) return CG_ERR_ALIGNMENT;
  cg::GenParams p = make_params(*desc, lay);
  return from_cuda(cg::launch_generate_propagating(p, gain, d_acts, d_refs, d_labels, d_ws, lay,
                                                   d_status, (cudaStream_t)stream));
}

cg_status cg_random_scores(uint64_t seed, uint32_t config_id0, uint32_t n_configs,
                           uint32_t n_canaries, uint32_t n_shards, float *d_scores,
                           cg_stream_t stream) {
  CG_TRACE("cg_random_scores");
  if (!d_scores || n_configs == 0 || n_canaries == 0 || n_shards == 0) return CG_ERR_INVALID_ARG;
  if ((uint64_t)config_id0 + n_configs > (1ull << 30)) return CG_ERR_INVALID_ARG;
  if (n_canaries > (1u << 24)) return CG_ERR_UNSUPPORTED;
  if ((uint64_t)n_configs * n_canaries * n_shards >= (1ull << 40)) return CG_ERR_UNSUPPORTED;
  if (!aligned(d_scores, 4)) return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_random_scores(seed, config_id0, n_configs, n_canaries, n_shards,
                                            d_scores, (cudaStream_t)stream));
}

cg_status cg_drift_workspace_size(uint32_t n_shards, uint32_t n_canaries, uint64_t seg_len,
                                  size_t *bytes) {
  if (!bytes || n_shards == 0 || n_canaries == 0 || seg_len == 0) return CG_ERR_INVALID_ARG;
  *bytes = cg::drift_ws_bytes((uint64_t)n_shards * n_canaries, seg_len);
  return CG_OK;
}

cg_status cg_drift_scores(const uint16_t *d_acts, const float *d_refs, uint32_t n_shards,
                          uint32_t n_canaries, uint64_t seg_len, float *d_scores,
                          uint64_t stat_stride, void *d_ws, size_t ws_bytes, int32_t *d_status,
                          cg_stream_t stream) {
  return cg_drift_scores_ex(d_acts, d_refs, n_shards, n_canaries, seg_len, d_scores, stat_stride,
                            d_ws, ws_bytes, d_status, CG_DRIFT_AUTO, stream);
}

cg_status cg_drift_scores_ex(const uint16_t *d_acts, const float *d_refs, uint32_t n_shards,
                             uint32_t n_canaries, uint64_t seg_len, float *d_scores,
                             uint64_t stat_stride, void *d_ws, size_t ws_bytes, int32_t *d_status,
                             int32_t algo, cg_stream_t stream) {
  CG_TRACE("cg_drift_scores_ex");
  return drift_scores_checked(d_acts, d_refs, 1, n_shards, n_canaries, seg_len, d_scores,
                              stat_stride, d_ws, ws_bytes, d_status, algo, stream);
}

cg_status cg_drift_scores_batch(const uint16_t *d_acts, const float *d_refs, uint32_t n_configs,
                                uint32_t n_shards, uint32_t n_canaries, uint64_t seg_len,
                                float *d_scores, uint64_t stat_stride, void *d_ws,
                                size_t ws_bytes, int32_t *d_status, cg_stream_t stream) {
  CG_TRACE("cg_drift_scores_batch");
  return drift_scores_checked(d_acts, d_refs, n_configs, n_shards, n_canaries, seg_len, d_scores,
                              stat_stride, d_ws, ws_bytes, d_status, CG_DRIFT_AUTO, stream);
}

cg_status cg_drift_scores_host(const uint16_t *h_acts, const float *d_refs, uint32_t n_shards,
                               uint32_t n_canaries, uint64_t seg_len, float *d_scores,
                               uint64_t stat_stride, void *d_ws, size_t ws_bytes,
                               int32_t *d_status, cg_stream_t stream) {
  CG_TRACE("cg_drift_scores_host");
  if (!h_acts) return CG_ERR_INVALID_ARG;
  // Only page-locked host memory registered with CUDA may be read by a
  // kernel; resolve its device-side address (equal to the host address
  // under unified addressing).
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, h_acts) != cudaSuccess) {
    cudaGetLastError();
    return CG_ERR_INVALID_ARG;
  }
  if (attr.type != cudaMemoryTypeHost || attr.devicePointer == nullptr) return CG_ERR_INVALID_ARG;
  return cg_drift_scores_ex(static_cast<const uint16_t *>(attr.devicePointer), d_refs, n_shards,
                            n_canaries, seg_len, d_scores, stat_stride, d_ws, ws_bytes, d_status,
                            CG_DRIFT_STREAM, stream);
}

cg_status cg_drift_scores_noalloc(const uint16_t *d_acts, const float *d_refs,
                                  uint32_t n_shards, uint32_t n_canaries, uint64_t seg_len,
                                  float *d_scores, uint64_t stat_stride, int32_t *d_status,
                                  cg_stream_t stream) {
  CG_TRACE("cg_drift_scores_noalloc");
  if (n_shards == 0 || n_canaries == 0 || seg_len == 0) return CG_ERR_INVALID_ARG;
  const uint64_t n_seg = (uint64_t)n_shards * n_canaries;
  if (seg_len > (1ull << 40) || n_seg > (1ull << 31)) return CG_ERR_UNSUPPORTED;
  if (n_seg * cg::drift_chunks_per_seg(seg_len) > CG_NOALLOC_MAX_WORK_ITEMS)
    return CG_ERR_UNSUPPORTED;
  if (!d_acts || !d_refs || !d_scores) return CG_ERR_INVALID_ARG;
  if (stat_stride < n_seg) return CG_ERR_INVALID_ARG;
  if (!aligned(d_acts, 16) || !aligned(d_refs, 16) || !aligned(d_scores, 4) ||
      (d_status && !aligned(d_status, 4)))
    return CG_ERR_ALIGNMENT;
  (void)d_status;   // the register-streaming kernel has no wait that could give up
  return from_cuda(cg::launch_drift_noalloc(d_acts, d_refs, n_shards, n_canaries, seg_len,
                                            d_scores, stat_stride, (cudaStream_t)stream));
}

cg_status cg_make_control_labels(const int8_t *d_labels, uint32_t n_configs,
                                 uint32_t n_canaries, uint32_t n_shards, uint64_t seed,
                                 uint32_t config_id0, int8_t *d_ctrl, int32_t *d_status,
                                 cg_stream_t stream) {
  CG_TRACE("cg_make_control_labels");
  if (!d_labels || !d_ctrl || n_configs == 0 || n_canaries == 0 || n_shards == 0)
    return CG_ERR_INVALID_ARG;
  if ((uint64_t)config_id0 + n_configs > (1ull << 30)) return CG_ERR_INVALID_ARG;
  if (n_canaries > (1u << 24)) return CG_ERR_UNSUPPORTED;
  if ((uint64_t)n_configs * n_canaries * n_shards >= (1ull << 40)) return CG_ERR_UNSUPPORTED;
  if (d_status && !aligned(d_status, 4)) return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_control_labels(d_labels, n_configs, n_canaries, n_shards, seed,
                                             config_id0, d_ctrl, d_status,
                                             (cudaStream_t)stream));
}

cg_status cg_auroc(const float *d_scores, const int8_t *d_labels, uint32_t n_configs,
                   uint32_t n_canaries, uint32_t n_shards, int64_t *d_u2, int64_t *d_gt,
                   int64_t *d_eq, double *d_auroc, int32_t *d_status, cg_stream_t stream) {
  CG_TRACE("cg_auroc");
  if (!d_scores || !d_labels || !d_u2 || !d_auroc || n_configs == 0 || n_canaries == 0 ||
      n_shards == 0)
    return CG_ERR_INVALID_ARG;
  if (n_shards > cg::kMaxRankShards) return CG_ERR_UNSUPPORTED;
  if ((uint64_t)n_configs * n_canaries * n_shards >= (1ull << 40)) return CG_ERR_UNSUPPORTED;
  if (!aligned(d_scores, 4) || !aligned(d_u2, 8) || !aligned(d_auroc, 8) ||
      (d_gt && !aligned(d_gt, 8)) || (d_eq && !aligned(d_eq, 8)) ||
      (d_status && !aligned(d_status, 4)))
    return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_auroc(d_scores, d_labels, n_configs, n_canaries, n_shards, d_u2,
                                    d_gt, d_eq, d_auroc, d_status, (cudaStream_t)stream));
}

cg_status cg_auroc_pooled(const float *d_scores, const int8_t *d_labels, uint32_t n_configs,
                          uint32_t n_canaries, uint32_t n_shards, int64_t *d_u2,
                          int64_t *d_n_mal, int64_t *d_n_ben, double *d_auroc, int32_t *d_status,
                          cg_stream_t stream) {
  CG_TRACE("cg_auroc_pooled");
  if (!d_scores || !d_labels || !d_u2 || !d_auroc || n_configs == 0 || n_canaries == 0 ||
      n_shards == 0)
    return CG_ERR_INVALID_ARG;
  if ((uint64_t)n_canaries * n_shards > cg::kMaxPooled) return CG_ERR_UNSUPPORTED;
  if ((uint64_t)n_configs * n_canaries * n_shards >= (1ull << 40)) return CG_ERR_UNSUPPORTED;
  if (!aligned(d_scores, 4) || !aligned(d_u2, 8) || !aligned(d_auroc, 8) ||
      (d_n_mal && !aligned(d_n_mal, 8)) || (d_n_ben && !aligned(d_n_ben, 8)) ||
      (d_status && !aligned(d_status, 4)))
    return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_auroc_pooled(d_scores, d_labels, n_configs, n_canaries, n_shards,
                                           d_u2, d_n_mal, d_n_ben, d_auroc, d_status,
                                           (cudaStream_t)stream));
}

cg_status cg_selftest_bounded_wait(uint32_t limit_us, int32_t *d_status, cg_stream_t stream) {
  CG_TRACE("cg_selftest_bounded_wait");
  if (!d_status || limit_us == 0 || limit_us > 10u * 1000u * 1000u) return CG_ERR_INVALID_ARG;
  if (!aligned(d_status, 4)) return CG_ERR_ALIGNMENT;
  return from_cuda(cg::launch_bounded_wait_probe(limit_us, d_status, (cudaStream_t)stream));
}

cg_status cg_read_status(const int32_t *d_status, cg_stream_t stream, int32_t *h_word) {
  CG_TRACE("cg_read_status");
  if (!d_status) return CG_ERR_INVALID_ARG;
  int32_t w = 0;
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e == cudaSuccess) e = cudaMemcpy(&w, d_status, sizeof(w), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return CG_ERR_CUDA;
  if (h_word) *h_word = w;
  if (w & CG_DEVFLAG_TIMEOUT) return CG_ERR_TIMEOUT;
  if (w & CG_DEVFLAG_NAN_SCORE) return CG_ERR_NAN_SCORE;
  if (w & CG_DEVFLAG_NO_BENIGN) return CG_ERR_NO_BENIGN;
  return CG_OK;
}

}  // extern "C"
