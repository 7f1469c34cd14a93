// auroc.cu -- the ranking test: exact Mann-Whitney counts per canary
// (Eq. 5, ties counted as one half) and their mean over canaries (Eq. 6),
// plus the labels of the scrambled-label negative control (Sec. 4.5).
//
// auroc_kernel: one block per configuration, one warp per canary at a time.
// For S <= 32 each lane holds one stage's score and label and the warp
// compares every (malicious, benign) pair through shuffles; larger S is
// strided over the lanes with the benign side read from global memory.
// Counts are integers (exact in any order); the configuration's A-hat is
// one fp64 division of exact integers when every canary has the same pair
// count, else the per-canary ratios added in canary order by one thread.
#include "cg_internal.h"
#include "cg_rng.cuh"

namespace cg {
namespace {

constexpr int kRankThreads = 256;
constexpr int kRankWarps = kRankThreads / 32;

__device__ __forceinline__ bool is_nan_f(float x) { return x != x; }

__global__ void __launch_bounds__(kRankThreads)
auroc_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels, uint32_t C,
             uint32_t N, uint32_t S, int64_t *__restrict__ u2_out, int64_t *__restrict__ gt_out,
             int64_t *__restrict__ eq_out, double *__restrict__ auroc, int32_t *status) {
  __shared__ long long warp_u2[kRankWarps];
  __shared__ long long warp_valid[kRankWarps];
  __shared__ long long warp_pairs[kRankWarps];   // common pair count seen by the warp, or -1
  __shared__ int warp_uniform[kRankWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
    long long my_u2 = 0, my_valid = 0, my_pairs = -1;
    int my_uniform = 1;
    bool saw_nan = false;
    for (uint32_t n = warp; n < N; n += kRankWarps) {
      const uint64_t base = ((uint64_t)c * N + n) * S;
      long long g = 0, e = 0;
      int nm = 0, nb = 0;
      if (S <= 32) {
        const bool in = (uint32_t)lane < S;
        const float m = in ? scores[base + lane] : 0.f;
        const int l = in ? (int)labels[base + lane] : -1;
        const bool labelled = (l == 0 || l == 1);
        if (labelled && is_nan_f(m)) saw_nan = true;
        int lg = 0, le = 0;
        for (uint32_t k = 0; k < S; ++k) {
          const float mk = __shfl_sync(0xFFFFFFFFu, m, k);
          const int lk = __shfl_sync(0xFFFFFFFFu, l, k);
          if (l == 1 && lk == 0) {
            lg += (m > mk);
            le += (m == mk);
          }
        }
        nm = __popc(__ballot_sync(0xFFFFFFFFu, l == 1));
        nb = __popc(__ballot_sync(0xFFFFFFFFu, l == 0));
        g = lg;
        e = le;
      } else {
        long long lg = 0, le = 0;
        int lm = 0, lb = 0;
        for (uint32_t i = lane; i < S; i += 32) {
          const float m = scores[base + i];
          const int l = (int)labels[base + i];
          if ((l == 0 || l == 1) && is_nan_f(m)) saw_nan = true;
          lm += (l == 1);
          lb += (l == 0);
          if (l != 1) continue;
          for (uint32_t j = 0; j < S; ++j) {
            if (labels[base + j] != 0) continue;
            const float mj = scores[base + j];
            lg += (m > mj);
            le += (m == mj);
          }
        }
        g = lg;
        e = le;
        nm = lm;
        nb = lb;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          nm += __shfl_xor_sync(0xFFFFFFFFu, nm, off);
          nb += __shfl_xor_sync(0xFFFFFFFFu, nb, off);
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        g += __shfl_xor_sync(0xFFFFFFFFu, g, off);
        e += __shfl_xor_sync(0xFFFFFFFFu, e, off);
      }
      if (lane == 0) {
        const uint64_t o = (uint64_t)c * N + n;
        const long long u2 = 2 * g + e;
        u2_out[o] = u2;
        if (gt_out) gt_out[o] = g;
        if (eq_out) eq_out[o] = e;
        const long long pairs = (long long)nm * nb;
        if (pairs > 0) {
          my_u2 += u2;
          my_valid += 1;
          if (my_pairs < 0) my_pairs = pairs;
          else if (my_pairs != pairs) my_uniform = 0;
        }
      }
    }
    if (__any_sync(0xFFFFFFFFu, saw_nan) && lane == 0 && status)
      atomicOr(status, CG_DEVFLAG_NAN_SCORE);
    if (lane == 0) {
      warp_u2[warp] = my_u2;
      warp_valid[warp] = my_valid;
      warp_pairs[warp] = my_pairs;
      warp_uniform[warp] = my_uniform;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      long long total = 0, valid = 0, common = -1;
      int uniform = 1;
      for (int w = 0; w < kRankWarps; ++w) {
        total += warp_u2[w];
        valid += warp_valid[w];
        uniform &= warp_uniform[w];
        if (warp_pairs[w] >= 0) {
          if (common < 0) common = warp_pairs[w];
          else if (common != warp_pairs[w]) uniform = 0;
        }
      }
      double A;
      if (valid == 0) {
        A = NAN;
      } else if (uniform) {
        A = __ddiv_rn((double)total, (double)(2 * common * valid));
      } else {
        // per-canary ratios in canary order (rare: pair counts differ)
        double acc = 0.0;
        for (uint32_t n = 0; n < N; ++n) {
          const uint64_t base = ((uint64_t)c * N + n) * S;
          long long nm = 0, nb = 0;
          for (uint32_t s = 0; s < S; ++s) {
            nm += (labels[base + s] == 1);
            nb += (labels[base + s] == 0);
          }
          if (nm * nb == 0) continue;
          acc = __dadd_rn(acc, __ddiv_rn((double)u2_out[(uint64_t)c * N + n], (double)(2 * nm * nb)));
        }
        A = __ddiv_rn(acc, (double)valid);
      }
      auroc[c] = A;
    }
    __syncthreads();
  }
}

// One thread per (configuration, canary): j* = the r-th benign stage in
// ascending order, r a bounded draw of aux stream (CONTROL, canary) with
// config id config_id0 + c; truly malicious stages are left out (-1).
__global__ void control_labels_kernel(const int8_t *__restrict__ labels, uint32_t C, uint32_t N,
                                      uint32_t S, uint64_t seed, uint32_t config_id0,
                                      int8_t *__restrict__ ctrl, int32_t *status) {
  const uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (uint64_t)C * N) return;
  const uint32_t c = (uint32_t)(t / N), n = (uint32_t)(t % N);
  const int8_t *l = labels + t * S;
  int8_t *o = ctrl + t * S;
  uint32_t b = 0;
  for (uint32_t s = 0; s < S; ++s) {
    const bool benign = (l[s] == 0);
    b += benign;
    o[s] = benign ? 0 : -1;
  }
  if (b == 0) {
    if (status) atomicOr(status, CG_DEVFLAG_NO_BENIGN);
    return;
  }
  AuxWords w = aux_words(seed, kAuxControl, n, config_id0 + c);
  bool gave_up = false;
  const uint32_t r = aux_bounded(w, b, &gave_up);
  if (gave_up && status) atomicOr(status, CG_DEVFLAG_TIMEOUT);
  uint32_t k = 0;
  for (uint32_t s = 0; s < S; ++s) {
    if (l[s] != 0) continue;
    if (k == r) {
      o[s] = 1;
      break;
    }
    ++k;
  }
}

}  // namespace

cudaError_t launch_auroc(const float *scores, const int8_t *labels, uint32_t C, uint32_t N,
                         uint32_t S, int64_t *u2, int64_t *gt, int64_t *eq, double *auroc,
                         int32_t *status, cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  uint64_t grid = (uint64_t)info.sm_count * 8;
  if (grid > C) grid = C;
  auroc_kernel<<<(unsigned)grid, kRankThreads, 0, stream>>>(scores, labels, C, N, S, u2, gt, eq,
                                                            auroc, status);
  return cudaGetLastError();
}

cudaError_t launch_control_labels(const int8_t *labels, uint32_t C, uint32_t N, uint32_t S,
                                  uint64_t seed, uint32_t config_id0, int8_t *ctrl,
                                  int32_t *status, cudaStream_t stream) {
  const uint64_t n = (uint64_t)C * N;
  control_labels_kernel<<<(unsigned)((n + 127) / 128), 128, 0, stream>>>(labels, C, N, S, seed,
                                                                         config_id0, ctrl, status);
  return cudaGetLastError();
}

}  // namespace cg
