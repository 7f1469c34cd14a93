/*
 * Plain C client of the canary_guard C ABI (no Python, no torch): generate
 * the tiny synthetic pipeline on the device, score every (stage, canary)
 * segment, draw the scrambled-label control and rank both label sets.
 * Then scores a batch of two configurations in one call (the first the
 * same pipeline) and the first configuration without a workspace, and
 * compares both with the single call.  Prints "A_hat <value> control
 * <value> status <code> batch_equal <0|1> noalloc_close <0|1>" and exits 0
 * on success.  Built and run by tests/test_gpu_c_client.py.
 */
#include <cuda_runtime_api.h>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "canary_guard.h"

#define CHECK_CG(x)                                                        \
  do {                                                                     \
    cg_status st_ = (x);                                                   \
    if (st_ != CG_OK) {                                                    \
      fprintf(stderr, "%s: %s\n", #x, cg_status_string(st_));              \
      return 1;                                                            \
    }                                                                      \
  } while (0)
#define CHECK_CUDA(x)                                                      \
  do {                                                                     \
    if ((x) != cudaSuccess) {                                              \
      fprintf(stderr, "%s failed\n", #x);                                  \
      return 1;                                                            \
    }                                                                      \
  } while (0)

int main(void) {
  const int32_t malicious[1] = {1};
  cg_pipeline_desc d = {0};
  d.n_shards = 4; d.hidden = 256; d.n_canaries = 16; d.tokens = 32;
  d.malicious = malicious; d.n_malicious = 1;
  d.noise = CG_NOISE_MULT; d.benign_sigma = 1e-3f; d.shard_sigma_lognormal = 0.f;
  d.n_outlier = 2; d.outlier_scale = 20.f;
  d.tamper = CG_TAMPER_ADDITIVE; d.tamper_param = 0.05f;
  d.seed = 0; d.config_id = 0;
  const size_t S = d.n_shards, N = d.n_canaries, L = (size_t)d.tokens * d.hidden;

  size_t gen_ws = 0, drift_ws = 0;
  CHECK_CG(cg_generate_workspace_size(&d, &gen_ws));
  CHECK_CG(cg_drift_workspace_size(d.n_shards, d.n_canaries, L, &drift_ws));

  uint16_t *acts; float *refs, *scores; int8_t *labels, *ctrl; void *gws, *dws;
  int64_t *u2; double *auroc; int32_t *status;
  CHECK_CUDA(cudaMalloc((void **)&acts, S * N * L * 2));
  CHECK_CUDA(cudaMalloc((void **)&refs, S * N * L * 4));
  CHECK_CUDA(cudaMalloc((void **)&scores, 3 * N * S * 4));
  CHECK_CUDA(cudaMalloc((void **)&labels, N * S));
  CHECK_CUDA(cudaMalloc((void **)&ctrl, N * S));
  CHECK_CUDA(cudaMalloc(&gws, gen_ws));
  CHECK_CUDA(cudaMalloc(&dws, drift_ws));
  CHECK_CUDA(cudaMalloc((void **)&u2, N * 8));
  CHECK_CUDA(cudaMalloc((void **)&auroc, 2 * 8));
  CHECK_CUDA(cudaMalloc((void **)&status, 4));
  CHECK_CUDA(cudaMemset(status, 0, 4));

  cg_stream_t stream = 0;
  CHECK_CG(cg_generate_pipeline(&d, acts, refs, labels, gws, gen_ws, status, stream));
  CHECK_CG(cg_drift_scores(acts, refs, d.n_shards, d.n_canaries, L, scores, N * S, dws, drift_ws,
                           status, stream));
  CHECK_CG(cg_make_control_labels(labels, 1, d.n_canaries, d.n_shards, 7, 0, ctrl, status,
                                  stream));
  CHECK_CG(cg_auroc(scores, labels, 1, d.n_canaries, d.n_shards, u2, NULL, NULL, auroc, status,
                    stream));
  CHECK_CG(cg_auroc(scores, ctrl, 1, d.n_canaries, d.n_shards, u2, NULL, NULL, auroc + 1, status,
                    stream));
  int32_t word = 0;
  cg_status st = cg_read_status(status, stream, &word);
  double a[2];
  CHECK_CUDA(cudaMemcpy(a, auroc, sizeof(a), cudaMemcpyDeviceToHost));

  /* a batch of two configurations: [2][S][N][L], the first this pipeline */
  uint16_t *acts2; float *refs2, *scores2, *scores3; void *dws2;
  size_t drift_ws2 = 0;
  CHECK_CG(cg_drift_workspace_size(2 * d.n_shards, d.n_canaries, L, &drift_ws2));
  CHECK_CUDA(cudaMalloc((void **)&acts2, 2 * S * N * L * 2));
  CHECK_CUDA(cudaMalloc((void **)&refs2, 2 * S * N * L * 4));
  CHECK_CUDA(cudaMalloc((void **)&scores2, 3 * 2 * N * S * 4));
  CHECK_CUDA(cudaMalloc((void **)&scores3, 3 * N * S * 4));
  CHECK_CUDA(cudaMalloc(&dws2, drift_ws2));
  cg_pipeline_desc d1 = d;
  d1.config_id = 1;
  CHECK_CG(cg_generate_pipeline(&d, acts2, refs2, NULL, gws, gen_ws, status, stream));
  CHECK_CG(cg_generate_pipeline(&d1, acts2 + S * N * L, refs2 + S * N * L, NULL, gws, gen_ws,
                                status, stream));
  CHECK_CG(cg_drift_scores_batch(acts2, refs2, 2, d.n_shards, d.n_canaries, L, scores2,
                                 2 * N * S, dws2, drift_ws2, status, stream));
  CHECK_CG(cg_drift_scores_noalloc(acts, refs, d.n_shards, d.n_canaries, L, scores3, N * S,
                                   status, stream));
  float one[3 * 16 * 4], two[3 * 2 * 16 * 4], na[3 * 16 * 4];
  CHECK_CUDA(cudaMemcpy(one, scores, sizeof(one), cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(two, scores2, sizeof(two), cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(na, scores3, sizeof(na), cudaMemcpyDeviceToHost));
  int batch_equal = 1, noalloc_close = 1;
  for (size_t k = 0; k < 3; ++k)
    for (size_t i = 0; i < N * S; ++i) {
      /* configuration 0 of the batch: the same bytes as the single call */
      if (memcmp(&one[k * N * S + i], &two[k * 2 * N * S + i], sizeof(float)) != 0)
        batch_equal = 0;
      /* the no-workspace call streams through registers: its fp32 sums are
         added in another order, so rel_l2 within 1e-5 relative, cos_dev
         within 1e-5 of max(cos_dev, rel_l2^2 / 2), max_abs exact */
      const float x = one[k * N * S + i], y = na[k * N * S + i], m = one[i];
      const float scale = k == 2 ? fmaxf(fabsf(x), 0.5f * m * m) : fabsf(x);
      if (k == 1 ? x != y : fabsf(x - y) > 1e-5f * scale + 1e-12f) noalloc_close = 0;
    }
  if (cg_read_status(status, stream, &word) != CG_OK) st = CG_ERR_TIMEOUT;
  printf("A_hat %.6f control %.6f status %d batch_equal %d noalloc_close %d\n", a[0], a[1],
         (int)st, batch_equal, noalloc_close);

  cudaFree(acts); cudaFree(refs); cudaFree(scores); cudaFree(labels); cudaFree(ctrl);
  cudaFree(gws); cudaFree(dws); cudaFree(u2); cudaFree(auroc); cudaFree(status);
  cudaFree(acts2); cudaFree(refs2); cudaFree(scores2); cudaFree(scores3); cudaFree(dws2);
  return (st == CG_OK && batch_equal && noalloc_close) ? 0 : 1;
}
