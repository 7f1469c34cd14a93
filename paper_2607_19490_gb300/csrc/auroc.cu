// auroc.cu -- the ranking test: exact Mann-Whitney counts per canary
// (Eq. 5, ties counted as one half) and their mean over canaries (Eq. 6),
// plus the labels of the scrambled-label negative control (Sec. 4.5).
//
// S <= 32: one lane per canary -- auroc_lane_config_kernel (many
// configurations: a warp per configuration), auroc_block_kernel (few
// configurations of at most 1024 canaries: a block per configuration, one
// launch) or auroc_lane_canary_kernel + auroc_config_kernel (few, more
// canaries: lanes over all canaries, then a combine).
// S > 32: one warp per canary with the stages strided over the lanes
// (auroc_kernel / auroc_canary_kernel).
// Counts are integers (exact in any order); the configuration's A-hat is
// one fp64 division of exact integers when every canary has the same pair
// count, else the per-canary ratios added in canary order by one thread.
#include <climits>

#include "cg_internal.h"
#include "cg_rng.cuh"

namespace cg {
namespace {

constexpr int kRankThreads = 256;
constexpr int kRankWarps = kRankThreads / 32;

__device__ __forceinline__ bool is_nan_f(float x) { return x != x; }

// A-hat of configuration c from its integer sums (Eq. 6): one fp64 division
// when every canary with a pair has the same pair count (pmin == pmax),
// else the per-canary ratios added in canary order; NaN without a pair.
__device__ double combine_auroc(const int8_t *__restrict__ labels, uint64_t c, uint32_t N,
                                uint32_t S, const int64_t *__restrict__ u2, long long total,
                                long long valid, long long pmin, long long pmax) {
  if (valid == 0) return NAN;
  if (pmin == pmax) return __ddiv_rn((double)total, (double)(2 * pmin * valid));
  double acc = 0.0;
  for (uint32_t n = 0; n < N; ++n) {
    const int8_t *l = labels + (c * N + n) * S;
    long long nm = 0, nb = 0;
    for (uint32_t s = 0; s < S; ++s) {
      nm += (l[s] == 1);
      nb += (l[s] == 0);
    }
    if (nm * nb == 0) continue;
    acc = __dadd_rn(acc, __ddiv_rn((double)u2[c * N + n], (double)(2 * nm * nb)));
  }
  return __ddiv_rn(acc, (double)valid);
}

__device__ __forceinline__ void canary_counts(const float *m_all, const int8_t *l_all, uint32_t S,
                                              int lane, long long &g, long long &e, int &nm,
                                              int &nb, bool &saw_nan) {
  g = 0;
  e = 0;
  if (S <= 32) {
    const bool in = (uint32_t)lane < S;
    const float m = in ? m_all[lane] : 0.f;
    const int l = in ? (int)l_all[lane] : -1;
    if ((l == 0 || l == 1) && is_nan_f(m)) saw_nan = true;
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
    int lm = 0, lb = 0;
    for (uint32_t i = lane; i < S; i += 32) {
      const float m = m_all[i];
      const int l = (int)l_all[i];
      if ((l == 0 || l == 1) && is_nan_f(m)) saw_nan = true;
      lm += (l == 1);
      lb += (l == 0);
      if (l != 1) continue;
      for (uint32_t j = 0; j < S; ++j) {
        if (l_all[j] != 0) continue;
        const float mj = m_all[j];
        g += (m > mj);
        e += (m == mj);
      }
    }
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
}

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
      long long g, e;
      int nm, nb;
      canary_counts(scores + base, labels + base, S, lane, g, e, nm, nb, saw_nan);
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

// Lane-per-canary ranking for S <= 32 (SP = S rounded up to 4, 8, 16 or
// 32): each lane loads its canary's scores and labels into registers
// (16-byte score loads and SP-byte label loads when the rows are exactly SP
// wide and aligned) and counts, for every malicious stage, the benign
// stages below it and equal to it.  A warp ranks 32 canaries at once with
// no cross-lane traffic.  Labels stay packed four to a word; the stage
// masks come from exact per-byte zero tests on the words.
template <int SP>
struct LaneRow {
  float m[SP];
  uint32_t lw[SP / 4];      // label bytes; 0xFF (excluded) beyond S
};

template <int SP>
__device__ __forceinline__ void lane_load(const float *__restrict__ scores,
                                          const int8_t *__restrict__ labels, uint64_t o,
                                          uint32_t S, bool vec, LaneRow<SP> &r) {
  const float *ms = scores + o * S;
  const int8_t *ls = labels + o * S;
  if (vec) {
#pragma unroll
    for (int k = 0; k < SP; k += 4) {
      const float4 v = *reinterpret_cast<const float4 *>(ms + k);
      r.m[k] = v.x; r.m[k + 1] = v.y; r.m[k + 2] = v.z; r.m[k + 3] = v.w;
    }
    if (SP == 4) {
      r.lw[0] = *reinterpret_cast<const uint32_t *>(ls);
    } else if (SP == 8) {
      const uint2 w = *reinterpret_cast<const uint2 *>(ls);
      r.lw[0] = w.x; r.lw[1 % (SP / 4)] = w.y;
    } else {
#pragma unroll
      for (int q = 0; q < SP / 16; ++q) {
        const uint4 w = reinterpret_cast<const uint4 *>(ls)[q];
        r.lw[(4 * q) % (SP / 4)] = w.x; r.lw[(4 * q + 1) % (SP / 4)] = w.y;
        r.lw[(4 * q + 2) % (SP / 4)] = w.z; r.lw[(4 * q + 3) % (SP / 4)] = w.w;
      }
    }
  } else {
#pragma unroll
    for (int w = 0; w < SP / 4; ++w) r.lw[w] = 0xFFFFFFFFu;
#pragma unroll
    for (int k = 0; k < SP; ++k) {
      const bool in = (uint32_t)k < S;
      r.m[k] = in ? ms[k] : 0.f;
      if (in) {
        const uint32_t sh = 8u * (k & 3);
        r.lw[k >> 2] = (r.lw[k >> 2] & ~(0xFFu << sh)) | ((uint32_t)(uint8_t)ls[k] << sh);
      }
    }
  }
}

// Stage masks keep stage k at bit 8 (k mod 4) + k / 4: label word w holds
// stages 4w .. 4w + 3 in its bytes, so its per-byte flags (bits 7, 15, 23,
// 31) land there with one right shift by 7 - w.  Every mask of a lane uses
// this order; only popcounts and ANDs combine them.
__host__ __device__ constexpr int stage_bit(int k) { return 8 * (k & 3) + (k >> 2); }

// Bit 8b + 7 of the result = (byte b of x == 0).  Per byte, the low seven
// bits plus 0x7F carry into bit 7 exactly when they are not all zero (no
// carry leaves the byte); OR-ing x adds the byte's own bit 7.
__device__ __forceinline__ uint32_t zero_byte_flags(uint32_t x) {
  return ~(((x & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | x) & 0x80808080u;
}

// The stage k whose mask bit is i (the inverse of stage_bit for S <= 32).
__device__ __forceinline__ int stage_of_bit(int i) { return 4 * (i & 7) + (i >> 3); }

// m[k] for a run-time k without dynamic register indexing: a tree of
// selects on the bits of k, low bit first (SP - 1 selects).
template <int SP>
__device__ __forceinline__ float select_stage(const float (&m)[SP], int k) {
  float t[SP];
#pragma unroll
  for (int j = 0; j < SP; ++j) t[j] = m[j];
#pragma unroll
  for (int half = SP / 2, bit = 0; half >= 1; half /= 2, ++bit) {
    const bool odd = (k >> bit) & 1;
#pragma unroll
    for (int j = 0; j < half; ++j) t[j] = odd ? t[2 * j + 1] : t[2 * j];
  }
  return t[0];
}

template <int SP>
__device__ __forceinline__ void lane_rank(const LaneRow<SP> &r, int &g, int &e, int &nm, int &nb,
                                          bool &saw_nan) {
  uint32_t mal = 0u, ben = 0u;
#pragma unroll
  for (int w = 0; w < SP / 4; ++w) {
    ben |= zero_byte_flags(r.lw[w]) >> (7 - w);                 // label 0
    mal |= zero_byte_flags(r.lw[w] ^ 0x01010101u) >> (7 - w);   // label 1
  }
  // a NaN anywhere in the row (one unordered compare per stage); only then
  // are the NaN stages matched against the labelled ones
  bool any_nan = false;
#pragma unroll
  for (int k = 0; k < SP; ++k) any_nan |= is_nan_f(r.m[k]);
  if (any_nan) {
    uint32_t nan = 0u;
#pragma unroll
    for (int k = 0; k < SP; ++k) nan |= (uint32_t)is_nan_f(r.m[k]) << stage_bit(k);
    if (nan & (mal | ben)) saw_nan = true;
  }
  nm = __popc(mal);
  nb = __popc(ben);
  int lg = 0, le = 0;
  // only the malicious stages are walked; m_i is picked by a select tree
  // and compared with every stage at once
  while (mal) {
    const int i = __ffs(mal) - 1;
    mal &= mal - 1u;
    const float mi = select_stage<SP>(r.m, stage_of_bit(i));
    uint32_t gtm = 0u, eqm = 0u;
#pragma unroll
    for (int j = 0; j < SP; ++j) {
      gtm |= (uint32_t)(mi > r.m[j]) << stage_bit(j);
      eqm |= (uint32_t)(mi == r.m[j]) << stage_bit(j);
    }
    lg += __popc(gtm & ben);
    le += __popc(eqm & ben);
  }
  g = lg;
  e = le;
}

template <int SP>
__device__ __forceinline__ void lane_counts(const float *__restrict__ scores,
                                            const int8_t *__restrict__ labels, uint64_t o,
                                            uint32_t S, bool vec, long long &g, long long &e,
                                            int &nm, int &nb, bool &saw_nan) {
  LaneRow<SP> r;
  lane_load<SP>(scores, labels, o, S, vec, r);
  int gi, ei;
  lane_rank<SP>(r, gi, ei, nm, nb, saw_nan);
  g = gi;
  e = ei;
}

template <int SP>
__global__ void __launch_bounds__(kRankThreads, SP <= 16 ? 4 : 2)
auroc_lane_config_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels,
                         uint32_t C, uint32_t N, uint32_t S, bool vec,
                         int64_t *__restrict__ u2_out, int64_t *__restrict__ gt_out,
                         int64_t *__restrict__ eq_out, double *__restrict__ auroc,
                         int32_t *status) {
  const int lane = threadIdx.x & 31;
  const uint64_t warps = (uint64_t)gridDim.x * kRankWarps;
  const bool narrow = (uint64_t)N * (SP * SP / 2) < (1ull << 32);
  bool saw_nan = false;
  for (uint64_t c = (uint64_t)blockIdx.x * kRankWarps + (threadIdx.x >> 5); c < C; c += warps) {
    // per-lane sums; 32-bit when no configuration total can reach 2^32
    // (a canary's 2U is at most 2 (SP/2)^2)
    uint32_t t32 = 0u, valid = 0u, pmin = 0xFFFFFFFFu, pmax = 0u;
    unsigned long long t64 = 0ull;
    auto record = [&](const LaneRow<SP> &r, uint64_t o) {
      int g, e, nm, nb;
      lane_rank<SP>(r, g, e, nm, nb, saw_nan);
      const uint32_t u2 = 2u * (uint32_t)g + (uint32_t)e;
      u2_out[o] = u2;
      if (gt_out) gt_out[o] = g;
      if (eq_out) eq_out[o] = e;
      const uint32_t pairs = (uint32_t)nm * (uint32_t)nb;
      if (pairs > 0) {
        if (narrow) t32 += u2;
        else t64 += u2;
        valid += 1u;
        pmin = min(pmin, pairs);
        pmax = max(pmax, pairs);
      }
    };
    // two canaries per lane per round, both loaded before either is ranked
    for (uint32_t n = lane; n < N; n += 64) {
      const uint64_t o = c * N + n;
      const bool two = n + 32 < N;
      LaneRow<SP> ra, rb;
      lane_load<SP>(scores, labels, o, S, vec, ra);
      if (two) lane_load<SP>(scores, labels, o + 32, S, vec, rb);
      record(ra, o);
      if (two) record(rb, o + 32);
    }
    valid = __reduce_add_sync(0xFFFFFFFFu, valid);
    pmin = __reduce_min_sync(0xFFFFFFFFu, pmin);
    pmax = __reduce_max_sync(0xFFFFFFFFu, pmax);
    long long total;
    if (narrow) {
      total = (long long)__reduce_add_sync(0xFFFFFFFFu, t32);
    } else {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) t64 += __shfl_xor_sync(0xFFFFFFFFu, t64, off);
      total = (long long)t64;
    }
    __syncwarp();   // every lane's u2 writes are visible to lane 0 below
    if (lane == 0)
      auroc[c] = combine_auroc(labels, c, N, S, u2_out, total, valid, pmin, pmax);
    __syncwarp();
  }
  if (__any_sync(0xFFFFFFFFu, saw_nan) && lane == 0 && status)
    atomicOr(status, CG_DEVFLAG_NAN_SCORE);
}

template <int SP>
__global__ void __launch_bounds__(kRankThreads)
auroc_lane_canary_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels,
                         uint64_t n_canaries_total, uint32_t S, bool vec,
                         int64_t *__restrict__ u2_out, int64_t *__restrict__ gt_out,
                         int64_t *__restrict__ eq_out, int32_t *status) {
  bool saw_nan = false;
  for (uint64_t o = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; o < n_canaries_total;
       o += (uint64_t)gridDim.x * blockDim.x) {
    long long g, e;
    int nm, nb;
    lane_counts<SP>(scores, labels, o, S, vec, g, e, nm, nb, saw_nan);
    u2_out[o] = 2 * g + e;
    if (gt_out) gt_out[o] = g;
    if (eq_out) eq_out[o] = e;
  }
  if (saw_nan && status) atomicOr(status, CG_DEVFLAG_NAN_SCORE);
}

// Few configurations of at most kBlockRankCanaries canaries: one block per
// configuration ranks its canaries (a thread per canary, lane_counts) and
// combines them itself, so a single-configuration call is one launch.
constexpr uint32_t kBlockRankCanaries = 1024;

template <int SP>
__global__ void __launch_bounds__(kRankThreads)
auroc_block_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels, uint32_t C,
                   uint32_t N, uint32_t S, bool vec, int64_t *__restrict__ u2_out,
                   int64_t *__restrict__ gt_out, int64_t *__restrict__ eq_out,
                   double *__restrict__ auroc, int32_t *status) {
  __shared__ unsigned long long red_total[kRankWarps];
  __shared__ uint32_t red_small[kRankWarps][3];   // valid, pmin, pmax
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  bool saw_nan = false;
  for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
    unsigned long long total = 0ull;
    uint32_t valid = 0u, pmin = 0xFFFFFFFFu, pmax = 0u;
    for (uint32_t n = tid; n < N; n += kRankThreads) {
      const uint64_t o = (uint64_t)c * N + n;
      long long g, e;
      int nm, nb;
      lane_counts<SP>(scores, labels, o, S, vec, g, e, nm, nb, saw_nan);
      const long long u2 = 2 * g + e;
      u2_out[o] = u2;
      if (gt_out) gt_out[o] = g;
      if (eq_out) eq_out[o] = e;
      const uint32_t pairs = (uint32_t)nm * (uint32_t)nb;
      if (pairs > 0) {
        total += (unsigned long long)u2;
        valid += 1u;
        pmin = min(pmin, pairs);
        pmax = max(pmax, pairs);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) total += __shfl_xor_sync(0xFFFFFFFFu, total, off);
    valid = __reduce_add_sync(0xFFFFFFFFu, valid);
    pmin = __reduce_min_sync(0xFFFFFFFFu, pmin);
    pmax = __reduce_max_sync(0xFFFFFFFFu, pmax);
    if (lane == 0) {
      red_total[warp] = total;
      red_small[warp][0] = valid;
      red_small[warp][1] = pmin;
      red_small[warp][2] = pmax;
    }
    __syncthreads();   // also makes every thread's u2 writes visible to thread 0
    if (tid == 0) {
      unsigned long long T = 0ull;
      uint32_t V = 0u, lo = 0xFFFFFFFFu, hi = 0u;
      for (int w = 0; w < kRankWarps; ++w) {
        T += red_total[w];
        V += red_small[w][0];
        lo = min(lo, red_small[w][1]);
        hi = max(hi, red_small[w][2]);
      }
      auroc[c] = combine_auroc(labels, c, N, S, u2_out, (long long)T, V, lo, hi);
    }
    __syncthreads();
  }
  if (__syncthreads_or(saw_nan) && tid == 0 && status) atomicOr(status, CG_DEVFLAG_NAN_SCORE);
}

// Small batches (few configurations): the same per-canary counts with one
// warp per (configuration, canary) across the whole grid, then one block
// per configuration combines them.  Integer sums make both paths give the
// same bits.
__global__ void __launch_bounds__(kRankThreads)
auroc_canary_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels,
                    uint64_t n_canaries_total, uint32_t S, int64_t *__restrict__ u2_out,
                    int64_t *__restrict__ gt_out, int64_t *__restrict__ eq_out, int32_t *status) {
  const int lane = threadIdx.x & 31;
  const uint64_t warps = (uint64_t)gridDim.x * kRankWarps;
  bool saw_nan = false;
  for (uint64_t o = (uint64_t)blockIdx.x * kRankWarps + (threadIdx.x >> 5); o < n_canaries_total;
       o += warps) {
    long long g, e;
    int nm, nb;
    canary_counts(scores + o * S, labels + o * S, S, lane, g, e, nm, nb, saw_nan);
    if (lane == 0) {
      u2_out[o] = 2 * g + e;
      if (gt_out) gt_out[o] = g;
      if (eq_out) eq_out[o] = e;
    }
  }
  if (__any_sync(0xFFFFFFFFu, saw_nan) && lane == 0 && status)
    atomicOr(status, CG_DEVFLAG_NAN_SCORE);
}

__global__ void __launch_bounds__(kRankThreads)
auroc_config_kernel(const int8_t *__restrict__ labels, uint32_t C, uint32_t N, uint32_t S,
                    const int64_t *__restrict__ u2, double *__restrict__ auroc) {
  __shared__ long long red[kRankWarps][4];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
    long long total = 0, valid = 0, pmin = LLONG_MAX, pmax = -1;
    for (uint32_t n = tid; n < N; n += kRankThreads) {
      const int8_t *l = labels + ((uint64_t)c * N + n) * S;
      long long nm = 0, nb = 0;
      for (uint32_t s = 0; s < S; ++s) {
        nm += (l[s] == 1);
        nb += (l[s] == 0);
      }
      const long long pairs = nm * nb;
      if (pairs > 0) {
        total += u2[(uint64_t)c * N + n];
        valid += 1;
        pmin = min(pmin, pairs);
        pmax = max(pmax, pairs);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      total += __shfl_down_sync(0xFFFFFFFFu, total, off);
      valid += __shfl_down_sync(0xFFFFFFFFu, valid, off);
      pmin = min(pmin, __shfl_down_sync(0xFFFFFFFFu, pmin, off));
      pmax = max(pmax, __shfl_down_sync(0xFFFFFFFFu, pmax, off));
    }
    if (lane == 0) {
      red[warp][0] = total;
      red[warp][1] = valid;
      red[warp][2] = pmin;
      red[warp][3] = pmax;
    }
    __syncthreads();
    if (tid == 0) {
      for (int w = 1; w < kRankWarps; ++w) {
        red[0][0] += red[w][0];
        red[0][1] += red[w][1];
        red[0][2] = min(red[0][2], red[w][2]);
        red[0][3] = max(red[0][3], red[w][3]);
      }
      const long long T = red[0][0], V = red[0][1];
      double A;
      if (V == 0) {
        A = NAN;
      } else if (red[0][2] == red[0][3]) {
        A = __ddiv_rn((double)T, (double)(2 * red[0][2] * V));
      } else {
        double acc = 0.0;
        for (uint32_t n = 0; n < N; ++n) {
          const int8_t *l = labels + ((uint64_t)c * N + n) * S;
          long long nm = 0, nb = 0;
          for (uint32_t s = 0; s < S; ++s) {
            nm += (l[s] == 1);
            nb += (l[s] == 0);
          }
          if (nm * nb == 0) continue;
          acc = __dadd_rn(acc, __ddiv_rn((double)u2[(uint64_t)c * N + n], (double)(2 * nm * nb)));
        }
        A = __ddiv_rn(acc, (double)V);
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

// ----------------------------------------------------------------- pooled
// Pooled Mann-Whitney over all canaries of a configuration.  One block per
// configuration: the labelled scores become 64-bit keys
// (order-preserving image of the float << 32 | label) in shared memory, a
// bitonic network sorts them, and every malicious key adds twice its
// midrank, lo + 1 + hi, where [lo, hi) is the run of its score found by
// binary search.  2U = sum(2 midrank) - n_mal (n_mal + 1), exact in int64.
constexpr int kPoolThreads = 256;
constexpr int kPoolWarps = kPoolThreads / 32;

__device__ __forceinline__ uint32_t order_key(float x) {
  uint32_t b = __float_as_uint(x);
  if (b == 0x80000000u) b = 0u;                         // -0 ranks with +0
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// First index of the sorted, padded k[0, M) (M a power of two; the padding
// key 0xFFFFFFFF is above every score's key) whose key is >= v (lower) or
// > v (upper): log2(M) fixed steps, no divergence.
__device__ __forceinline__ uint32_t bound_u32(const uint32_t *k, uint32_t M, uint32_t v,
                                              bool upper) {
  uint32_t pos = 0;
  for (uint32_t step = M >> 1; step > 0; step >>= 1) {
    const uint32_t x = k[pos + step - 1];
    pos += (upper ? (x <= v) : (x < v)) ? step : 0u;
  }
  const uint32_t x = k[pos];
  return pos + ((upper ? (x <= v) : (x < v)) ? 1u : 0u);
}

// Bitonic sort of up to 64 keys held by one warp, two per lane (key e at
// register e / 32 of lane e % 32): stride 32 swaps the lane's registers,
// smaller strides pair lanes through shuffles.
__device__ __forceinline__ void warp_sort64(uint32_t &r0, uint32_t &r1, uint32_t M, int lane) {
  for (uint32_t k = 2; k <= M; k <<= 1) {
    for (uint32_t j = k >> 1; j > 0; j >>= 1) {
      if (j == 32) {
        const bool up = ((uint32_t)lane & k) == 0;          // e = lane, partner lane + 32
        const uint32_t lo = min(r0, r1), hi = max(r0, r1);
        r0 = up ? lo : hi;
        r1 = up ? hi : lo;
      } else {
        const uint32_t p0 = __shfl_xor_sync(0xFFFFFFFFu, r0, (int)j);
        const uint32_t p1 = __shfl_xor_sync(0xFFFFFFFFu, r1, (int)j);
        const bool lower = ((uint32_t)lane & j) == 0;
        const bool up0 = ((uint32_t)lane & k) == 0;
        const bool up1 = (((uint32_t)lane + 32u) & k) == 0;
        r0 = (lower == up0) ? min(r0, p0) : max(r0, p0);
        r1 = (lower == up1) ? min(r1, p1) : max(r1, p1);
      }
    }
  }
}

// Pooled Mann-Whitney (Sec. 3.4), one block per configuration.  The
// labelled scores become order-preserving 32-bit keys, compacted into
// shared memory (malicious from the front, benign from the back, warp-
// aggregated offsets; the order inside each side does not matter).  Only
// the smaller side is sorted (a block bitonic sort of its padded
// power-of-two size Ms); every key of the larger side then takes its lower
// and upper bound in the sorted side, which give its pairs above and tied:
//   smaller side malicious: gt += #(m > b) = s - upper(b), eq += upper - lower
//   smaller side benign:    gt += #(b < m) = lower(m),     eq += upper - lower
// 2U = 2 gt + eq is an exact integer and A-hat = 2U / (2 n_m n_b) one fp64
// division.  Shared memory: per + Ms 32-bit keys.
__global__ void __launch_bounds__(kPoolThreads)
auroc_pooled_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels,
                    uint32_t C, uint32_t per, uint32_t Ms, int64_t *__restrict__ u2_out,
                    int64_t *__restrict__ nm_out, int64_t *__restrict__ nb_out,
                    double *__restrict__ auroc, int32_t *status) {
  extern __shared__ uint32_t pool_keys[];
  uint32_t *sorted = pool_keys + per;
  __shared__ unsigned int n_mal_s, n_ben_s;
  __shared__ unsigned long long red[kPoolWarps][2];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t lt_mask = (1u << lane) - 1u;
  bool nan_seen = false;
  for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
    if (tid == 0) n_mal_s = n_ben_s = 0u;
    __syncthreads();
    const float *m = scores + (uint64_t)c * per;
    const int8_t *l = labels + (uint64_t)c * per;
    for (uint32_t i0 = 0; i0 < per; i0 += kPoolThreads) {
      const uint32_t i = i0 + tid;
      int lab = -1;
      float x = 0.f;
      if (i < per) {
        lab = l[i];
        if (lab == 0 || lab == 1) {
          x = m[i];
          if (is_nan_f(x)) {
            nan_seen = true;
            lab = -1;
          }
        }
      }
      const uint32_t mal = __ballot_sync(0xFFFFFFFFu, lab == 1);
      const uint32_t ben = __ballot_sync(0xFFFFFFFFu, lab == 0);
      uint32_t base_m = 0u, base_b = 0u;
      if (lane == 0) {
        if (mal) base_m = atomicAdd(&n_mal_s, (unsigned)__popc(mal));
        if (ben) base_b = atomicAdd(&n_ben_s, (unsigned)__popc(ben));
      }
      base_m = __shfl_sync(0xFFFFFFFFu, base_m, 0);
      base_b = __shfl_sync(0xFFFFFFFFu, base_b, 0);
      if (lab == 1) pool_keys[base_m + __popc(mal & lt_mask)] = order_key(x);
      else if (lab == 0) pool_keys[per - 1u - (base_b + __popc(ben & lt_mask))] = order_key(x);
    }
    __syncthreads();
    const uint32_t nm = n_mal_s, nb = n_ben_s;
    const bool small_mal = nm <= nb;
    const uint32_t ns = small_mal ? nm : nb, nl = small_mal ? nb : nm;
    const uint32_t *small = small_mal ? pool_keys : pool_keys + (per - nb);
    const uint32_t *large = small_mal ? pool_keys + (per - nb) : pool_keys;
    uint32_t M = 1;
    while (M < ns) M <<= 1;
    if (M <= 64) {
      // a small side of up to 64 keys: one warp sorts it in registers
      if (warp == 0) {
        uint32_t r0 = (uint32_t)lane < ns ? small[lane] : 0xFFFFFFFFu;
        uint32_t r1 = (uint32_t)lane + 32u < ns ? small[lane + 32] : 0xFFFFFFFFu;
        warp_sort64(r0, r1, M, lane);
        if ((uint32_t)lane < M) sorted[lane] = r0;
        if ((uint32_t)lane + 32u < M) sorted[lane + 32] = r1;
      }
      __syncthreads();
    } else {
      for (uint32_t i = tid; i < M; i += kPoolThreads) sorted[i] = i < ns ? small[i] : 0xFFFFFFFFu;
      __syncthreads();
      for (uint32_t k = 2; k <= M; k <<= 1) {
        for (uint32_t j = k >> 1; j > 0; j >>= 1) {
          for (uint32_t i = tid; i < M; i += kPoolThreads) {
            const uint32_t ixj = i ^ j;
            if (ixj > i) {
              const uint32_t a = sorted[i], b = sorted[ixj];
              if ((a > b) == ((i & k) == 0)) {
                sorted[i] = b;
                sorted[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      }
    }
    unsigned long long gt = 0ull, eq = 0ull;
    if (ns > 0) {
      for (uint32_t i = tid; i < nl; i += kPoolThreads) {
        const uint32_t v = large[i];
        const uint32_t lo = bound_u32(sorted, M, v, false);
        const uint32_t hi = bound_u32(sorted, M, v, true);
        gt += small_mal ? (ns - hi) : lo;
        eq += hi - lo;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      gt += __shfl_down_sync(0xFFFFFFFFu, gt, off);
      eq += __shfl_down_sync(0xFFFFFFFFu, eq, off);
    }
    if (lane == 0) {
      red[warp][0] = gt;
      red[warp][1] = eq;
    }
    __syncthreads();
    if (tid == 0) {
      unsigned long long G = 0ull, E = 0ull;
      for (int w = 0; w < kPoolWarps; ++w) {
        G += red[w][0];
        E += red[w][1];
      }
      const long long u2 = (long long)(2ull * G + E);
      const long long NM = nm, NB = nb;
      u2_out[c] = u2;
      if (nm_out) nm_out[c] = NM;
      if (nb_out) nb_out[c] = NB;
      auroc[c] = (NM * NB > 0) ? __ddiv_rn((double)u2, (double)(2 * NM * NB)) : NAN;
    }
    __syncthreads();
  }
  if (__any_sync(0xFFFFFFFFu, nan_seen) && lane == 0 && status)
    atomicOr(status, CG_DEVFLAG_NAN_SCORE);
}

// Pairs of the larger side against the sorted, padded smaller side of
// M = 2^LOG keys: for each larger-side key v (lane-strided), the lower and
// upper bounds of v in `sorted` by LOG unrolled halving steps each, both
// searches interleaved; gt and eq as in auroc_pooled_kernel.
template <int LOG>
__device__ __forceinline__ void pool_count(const uint32_t *sorted, const uint32_t *large,
                                           uint32_t nl, uint32_t ns, bool small_mal, int lane,
                                           uint32_t &gt, uint32_t &eq) {
  for (uint32_t i = lane; i < nl; i += 32) {
    const uint32_t v = large[i];
    uint32_t pl = 0u, ph = 0u;
#pragma unroll
    for (int b = LOG - 1; b >= 0; --b) {
      const uint32_t step = 1u << b;
      const uint32_t xl = sorted[pl + step - 1], xh = sorted[ph + step - 1];
      pl += (xl < v) ? step : 0u;
      ph += (xh <= v) ? step : 0u;
    }
    const uint32_t lo = pl + (sorted[pl] < v ? 1u : 0u);
    const uint32_t hi = ph + (sorted[ph] <= v ? 1u : 0u);
    gt += small_mal ? (ns - hi) : lo;
    eq += hi - lo;
  }
}

// Pooled Mann-Whitney with one warp per configuration, for configurations
// of at most kPoolWarpMaxPer scores: the same compaction, sort of the
// smaller side and bound searches as auroc_pooled_kernel, but each warp
// works in its own part of shared memory and synchronises only itself, so
// the eight warps of a block rank eight configurations at once with no
// block-wide barrier and no shared atomics.  The smaller side holds at most
// per / 2 keys: up to 64 they are sorted in registers (warp_sort64), above
// that by a warp bitonic sort in shared memory.  Counts fit 32 bits
// (n_mal n_ben <= 512^2).
constexpr uint32_t kPoolWarpMaxPer = 1024;
constexpr uint32_t kPoolWarpMaxSmall = kPoolWarpMaxPer / 2;
constexpr size_t kPoolWarpSmem = (size_t)kPoolWarps * (kPoolWarpMaxPer + kPoolWarpMaxSmall) * 4;

__global__ void __launch_bounds__(kPoolThreads)
auroc_pooled_warp_kernel(const float *__restrict__ scores, const int8_t *__restrict__ labels,
                         uint32_t C, uint32_t per, bool vec, int64_t *__restrict__ u2_out,
                         int64_t *__restrict__ nm_out, int64_t *__restrict__ nb_out,
                         double *__restrict__ auroc, int32_t *status) {
  extern __shared__ uint32_t pw_smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t *keys = pw_smem + (size_t)warp * (kPoolWarpMaxPer + kPoolWarpMaxSmall);
  uint32_t *sorted = keys + kPoolWarpMaxPer;
  const uint32_t lt_mask = (1u << lane) - 1u;
  bool nan_seen = false;
  const uint64_t warps = (uint64_t)gridDim.x * kPoolWarps;
  for (uint64_t c = (uint64_t)blockIdx.x * kPoolWarps + warp; c < C; c += warps) {
    const float *m = scores + c * per;
    const int8_t *l = labels + c * per;
    // labelled scores -> order-preserving keys: malicious from the front,
    // benign from the back (the order inside each side does not matter)
    uint32_t nm = 0u, nb = 0u;                       // warp-uniform counts so far
    auto place = [&](int lab, float x) {
      if (lab == 0 || lab == 1) {
        if (is_nan_f(x)) {
          nan_seen = true;
          lab = -1;
        }
      } else {
        lab = -1;
      }
      const uint32_t mal = __ballot_sync(0xFFFFFFFFu, lab == 1);
      const uint32_t ben = __ballot_sync(0xFFFFFFFFu, lab == 0);
      if (lab == 1) keys[nm + __popc(mal & lt_mask)] = order_key(x);
      else if (lab == 0) keys[per - 1u - (nb + __popc(ben & lt_mask))] = order_key(x);
      nm += __popc(mal);
      nb += __popc(ben);
    };
    if (vec) {
      // 4 scores (16 bytes) and 4 labels (4 bytes) per lane and load, 4 loads
      // of each in flight before any is placed
      constexpr int U = 4;
      for (uint32_t i0 = 0; i0 < per; i0 += 128u * U) {
        float4 xv[U];
        uint32_t lv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const uint32_t i = i0 + 128u * u + 4u * (uint32_t)lane;
          if (i < per) {
            xv[u] = *reinterpret_cast<const float4 *>(m + i);
            lv[u] = *reinterpret_cast<const uint32_t *>(l + i);
          } else {
            xv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
            lv[u] = 0xFFFFFFFFu;                     // -1: left out
          }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          place((int)(int8_t)(lv[u] & 0xFFu), xv[u].x);
          place((int)(int8_t)((lv[u] >> 8) & 0xFFu), xv[u].y);
          place((int)(int8_t)((lv[u] >> 16) & 0xFFu), xv[u].z);
          place((int)(int8_t)(lv[u] >> 24), xv[u].w);
        }
      }
    } else {
      for (uint32_t i0 = 0; i0 < per; i0 += 32) {
        const uint32_t i = i0 + (uint32_t)lane;
        int lab = -1;
        float x = 0.f;
        if (i < per) {
          lab = l[i];
          if (lab == 0 || lab == 1) x = m[i];
        }
        place(lab, x);
      }
    }
    __syncwarp();
    const bool small_mal = nm <= nb;
    const uint32_t ns = small_mal ? nm : nb, nl = small_mal ? nb : nm;
    const uint32_t *small = small_mal ? keys : keys + (per - nb);
    const uint32_t *large = small_mal ? keys + (per - nb) : keys;
    uint32_t M = 1;
    while (M < ns) M <<= 1;
    if (M <= 64) {
      uint32_t r0 = (uint32_t)lane < ns ? small[lane] : 0xFFFFFFFFu;
      uint32_t r1 = (uint32_t)lane + 32u < ns ? small[lane + 32] : 0xFFFFFFFFu;
      warp_sort64(r0, r1, M, lane);
      if ((uint32_t)lane < M) sorted[lane] = r0;
      if ((uint32_t)lane + 32u < M) sorted[lane + 32] = r1;
    } else {
      for (uint32_t i = lane; i < M; i += 32) sorted[i] = i < ns ? small[i] : 0xFFFFFFFFu;
      __syncwarp();
      for (uint32_t k = 2; k <= M; k <<= 1) {
        for (uint32_t j = k >> 1; j > 0; j >>= 1) {
          for (uint32_t i = lane; i < M; i += 32) {
            const uint32_t ixj = i ^ j;
            if (ixj > i) {
              const uint32_t a = sorted[i], b = sorted[ixj];
              if ((a > b) == ((i & k) == 0)) {
                sorted[i] = b;
                sorted[ixj] = a;
              }
            }
          }
          __syncwarp();
        }
      }
    }
    __syncwarp();
    uint32_t gt = 0u, eq = 0u;
    if (ns > 0) {
      switch (31 - __clz(M)) {                      // log2 M, 0 .. 9
        case 0: pool_count<0>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 1: pool_count<1>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 2: pool_count<2>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 3: pool_count<3>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 4: pool_count<4>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 5: pool_count<5>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 6: pool_count<6>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 7: pool_count<7>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        case 8: pool_count<8>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
        default: pool_count<9>(sorted, large, nl, ns, small_mal, lane, gt, eq); break;
      }
    }
    gt = __reduce_add_sync(0xFFFFFFFFu, gt);
    eq = __reduce_add_sync(0xFFFFFFFFu, eq);
    if (lane == 0) {
      const long long u2 = 2ll * (long long)gt + (long long)eq;
      const long long NM = nm, NB = nb;
      u2_out[c] = u2;
      if (nm_out) nm_out[c] = NM;
      if (nb_out) nb_out[c] = NB;
      auroc[c] = (NM * NB > 0) ? __ddiv_rn((double)u2, (double)(2 * NM * NB)) : NAN;
    }
    __syncwarp();   // keys and sorted are rewritten by the next configuration
  }
  if (__any_sync(0xFFFFFFFFu, nan_seen) && lane == 0 && status)
    atomicOr(status, CG_DEVFLAG_NAN_SCORE);
}

}  // namespace

cudaError_t launch_auroc_pooled(const float *scores, const int8_t *labels, uint32_t C,
                                uint32_t N, uint32_t S, int64_t *u2, int64_t *n_mal,
                                int64_t *n_ben, double *auroc, int32_t *status,
                                cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  const uint32_t per = N * S;
  if (per <= kPoolWarpMaxPer) {
    // a warp per configuration, eight per block, the blocks that fit at once
    uint64_t grid = ((uint64_t)C + kPoolWarps - 1) / kPoolWarps;
    int occ = 0;
    cudaError_t err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &occ, auroc_pooled_warp_kernel, kPoolThreads, kPoolWarpSmem);
    if (err != cudaSuccess) return err;
    const uint64_t resident = (uint64_t)info.sm_count * (uint64_t)(occ > 0 ? occ : 1);
    if (grid > resident) grid = resident;
    // 16-byte score and 4-byte label loads when every configuration's row
    // starts on those boundaries
    const bool vec = (per % 4) == 0 && ((uintptr_t)scores % 16) == 0 &&
                     ((uintptr_t)labels % 4) == 0;
    auroc_pooled_warp_kernel<<<(unsigned)grid, kPoolThreads, kPoolWarpSmem, stream>>>(
        scores, labels, C, per, vec, u2, n_mal, n_ben, auroc, status);
    return cudaGetLastError();
  }
  uint32_t Ms = 1;                                // the smaller side holds at most per / 2 keys
  while (Ms < (per + 1) / 2) Ms <<= 1;
  const size_t smem = (size_t)(per + Ms) * sizeof(uint32_t);
  cudaError_t err = cudaFuncSetAttribute(auroc_pooled_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  uint64_t grid = C;
  if (C > (uint32_t)info.sm_count) {
    int occ = 0;
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, auroc_pooled_kernel, kPoolThreads,
                                                        smem);
    if (err != cudaSuccess) return err;
    const uint64_t resident = (uint64_t)info.sm_count * (uint64_t)(occ > 0 ? occ : 1);
    if (grid > resident) grid = resident;
  }
  auroc_pooled_kernel<<<(unsigned)grid, kPoolThreads, smem, stream>>>(scores, labels, C, per, Ms,
                                                                      u2, n_mal, n_ben, auroc,
                                                                      status);
  return cudaGetLastError();
}

cudaError_t launch_auroc(const float *scores, const int8_t *labels, uint32_t C, uint32_t N,
                         uint32_t S, int64_t *u2, int64_t *gt, int64_t *eq, double *auroc,
                         int32_t *status, cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  const bool many = (uint64_t)C >= 2ull * (uint64_t)info.sm_count;
  // S <= 32: a warp per configuration pays off from about 8 configurations
  // per SM; below that a block per configuration finishes sooner (324
  // configurations x 64 canaries: 5.6 us against 6.5 us, kernels alone)
  const bool many_lane = (uint64_t)C >= 8ull * (uint64_t)info.sm_count;
  const uint64_t total = (uint64_t)C * N;
  const uint64_t cap = (uint64_t)info.sm_count * 8;
  if (S > 32) {
    // wide pipelines: one warp per canary, stages strided over the lanes
    if (many) {
      const uint64_t grid = cap < C ? cap : C;
      auroc_kernel<<<(unsigned)grid, kRankThreads, 0, stream>>>(scores, labels, C, N, S, u2, gt,
                                                                eq, auroc, status);
      return cudaGetLastError();
    }
    uint64_t blocks = (total + kRankWarps - 1) / kRankWarps;
    if (blocks > cap) blocks = cap;
    auroc_canary_kernel<<<(unsigned)blocks, kRankThreads, 0, stream>>>(scores, labels, total, S, u2,
                                                                       gt, eq, status);
  } else {
    const int SP = S <= 4 ? 4 : S <= 8 ? 8 : S <= 16 ? 16 : 32;
    // 16-byte row loads only when a row is exactly SP scores and 16-byte aligned
    const bool vec = (S == (uint32_t)SP) && ((uintptr_t)scores % 16 == 0) &&
                     ((uintptr_t)labels % (SP < 16 ? SP : 16) == 0);
    if (many_lane) {
      const uint64_t grid = ((uint64_t)C + kRankWarps - 1) / kRankWarps;   // a warp each
#define CG_LANE_CONFIG(P)                                                                     \
  auroc_lane_config_kernel<P><<<(unsigned)grid, kRankThreads, 0, stream>>>(scores, labels, C, N, \
                                                                         S, vec, u2, gt, eq,   \
                                                                         auroc, status)
      switch (SP) {
        case 4: CG_LANE_CONFIG(4); break;
        case 8: CG_LANE_CONFIG(8); break;
        case 16: CG_LANE_CONFIG(16); break;
        default: CG_LANE_CONFIG(32); break;
      }
#undef CG_LANE_CONFIG
      return cudaGetLastError();
    }
    if (N <= kBlockRankCanaries) {
      // few configurations of few canaries: one block each, one launch
#define CG_BLOCK_RANK(P)                                                                     \
  auroc_block_kernel<P><<<C, kRankThreads, 0, stream>>>(scores, labels, C, N, S, vec, u2, gt, eq, \
                                                       auroc, status)
      switch (SP) {
        case 4: CG_BLOCK_RANK(4); break;
        case 8: CG_BLOCK_RANK(8); break;
        case 16: CG_BLOCK_RANK(16); break;
        default: CG_BLOCK_RANK(32); break;
      }
#undef CG_BLOCK_RANK
      return cudaGetLastError();
    }
    uint64_t blocks = (total + kRankThreads - 1) / kRankThreads;
    if (blocks > cap) blocks = cap;
#define CG_LANE_CANARY(P)                                                                   \
  auroc_lane_canary_kernel<P><<<(unsigned)blocks, kRankThreads, 0, stream>>>(scores, labels, \
                                                                           total, S, vec, u2, \
                                                                           gt, eq, status)
    switch (SP) {
      case 4: CG_LANE_CANARY(4); break;
      case 8: CG_LANE_CANARY(8); break;
      case 16: CG_LANE_CANARY(16); break;
      default: CG_LANE_CANARY(32); break;
    }
#undef CG_LANE_CANARY
  }
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  auroc_config_kernel<<<C, kRankThreads, 0, stream>>>(labels, C, N, S, u2, auroc);
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
