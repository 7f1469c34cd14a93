/*
 * Plain C client of the canary_guard C ABI (no Python, no torch): generate
 * the tiny synthetic pipeline on the device, score every (stage, canary)
 * segment, draw the scrambled-label control and rank both label sets.
 * Prints "A_hat <value> control <value> status <code>" and exits 0 on
 * success.  Built and run by tests/test_gpu_c_client.py.
 */
#include <cuda_runtime_api.h>
#include <stdint.h>
#include <stdio.h>

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
  printf("A_hat %.6f control %.6f status %d\n", a[0], a[1], (int)st);

  cudaFree(acts); cudaFree(refs); cudaFree(scores); cudaFree(labels); cudaFree(ctrl);
  cudaFree(gws); cudaFree(dws); cudaFree(u2); cudaFree(auroc); cudaFree(status);
  return st == CG_OK ? 0 : 1;
}
