// generate.cu -- device-side synthetic pipeline (Eq. 1-3 stand-in, Sec. 3.3).
//
// Materialises, for one configuration, the fp32 hop references and the fp16
// live activations of every (stage, canary) segment, plus the labels:
//   gen_setup_kernel    per-configuration draws: outlier-channel mask,
//                       per-stage sigma (lognormal spread), flipped-channel
//                       masks of the malicious stages; labels [N][S]
//   gen_refs_kernel     pass 1: reference normals -> fp32 references.  A
//                       segment whose live values follow element by element
//                       (benign a (1 + sigma_s z), sign flips, rescale) gets
//                       its fp16 live values here too, from the registers.
//                       The other segments get the sums their live values
//                       depend on: sum |a| (Eq. 2: mu = ||a||_1 / (T d)) for
//                       benign stages under the Eq. 2 noise model; sum a^2
//                       and sum g^2 (the Gaussian tamper's ||v|| and ||g||)
//   gen_coef_kernel     per-segment scalar from those sums (fixed order, fp64)
//   gen_live_kernel     pass 2, only for those segments: references read
//                       back, noise or tamper normals drawn, fp16 live
//                       values stored
// Random draws follow the counter layout of cg_rng.cuh: element e of
// segment seg on stream k uses block e / 4 of counter
// (e / 4, seg, 4 config_id + k, 0).
#include <cuda_fp16.h>

#include "cg_internal.h"
#include "cg_rng.cuh"

namespace cg {
namespace {

__device__ __forceinline__ bool mask_bit(const uint32_t *mask, uint32_t c) {
  return (__ldg(mask + (c >> 5)) >> (c & 31)) & 1u;
}

__device__ __forceinline__ bool is_malicious(const GenParams &p, uint32_t s) {
  return (p.mal_bits[s >> 5] >> (s & 31)) & 1u;
}

// ----------------------------------------------------------------- setup
// One block.  Threads first clear the masks; then thread 0 draws the
// outlier channels, one thread per stage draws its sigma, and one thread per
// malicious stage draws its flipped channels (each writes only its own mask
// row).  Distinct values come from successive bounded draws with duplicates
// redrawn; the draw count is capped and a cap hit is reported.
__global__ void gen_setup_kernel(GenParams p, uint32_t *outlier_mask, uint32_t *flip_mask,
                                 float *stage_sigma, int8_t *labels, int32_t *status) {
  const int tid = threadIdx.x;
  for (uint32_t i = tid; i < p.mask_words; i += blockDim.x) outlier_mask[i] = 0u;
  for (uint64_t i = tid; i < (uint64_t)p.S * p.mask_words; i += blockDim.x) flip_mask[i] = 0u;
  __syncthreads();
  bool gave_up = false;
  if (tid == 0 && p.n_outlier > 0) {
    AuxWords w = aux_words(p.seed, kAuxOutlier, 0, p.config_id);
    uint32_t got = 0;
    const uint64_t cap = 64ull * p.d + 1024;
    for (uint64_t tries = 0; got < p.n_outlier; ++tries) {
      if (tries >= cap) { gave_up = true; break; }
      const uint32_t c = aux_bounded(w, p.d, &gave_up);
      const uint32_t bit = 1u << (c & 31);
      if (outlier_mask[c >> 5] & bit) continue;
      outlier_mask[c >> 5] |= bit;
      ++got;
    }
  }
  for (uint32_t s = tid; s < p.S; s += blockDim.x) {
    float sig = p.sigma;
    if (p.lognormal > 0.f) {
      AuxWords w = aux_words(p.seed, kAuxStageSigma, s, p.config_id);
      const uint32_t x0 = aux_next(w), x1 = aux_next(w);
      sig = p.sigma * expf(p.lognormal * box_muller(x0, x1).x);
    }
    stage_sigma[s] = sig;
    if (p.tamper == CG_TAMPER_SIGNFLIP_CHANNELS && is_malicious(p, s)) {
      uint32_t *row = flip_mask + (uint64_t)s * p.mask_words;
      AuxWords w = aux_words(p.seed, kAuxFlip, s, p.config_id);
      uint32_t got = 0;
      const uint64_t cap = 64ull * p.d + 1024;
      for (uint64_t tries = 0; got < p.n_flip; ++tries) {
        if (tries >= cap) { gave_up = true; break; }
        const uint32_t c = aux_bounded(w, p.d, &gave_up);
        const uint32_t bit = 1u << (c & 31);
        if (row[c >> 5] & bit) continue;
        row[c >> 5] |= bit;
        ++got;
      }
    }
  }
  if (labels) {
    for (uint64_t i = tid; i < (uint64_t)p.N * p.S; i += blockDim.x)
      labels[i] = is_malicious(p, (uint32_t)(i % p.S)) ? 1 : 0;
  }
  if (gave_up && status) atomicOr(status, CG_DEVFLAG_TIMEOUT);
}

// The eight normals of elements e0 .. e0 + 7 (blocks q0 = e0 / 4 and q0 + 1
// of counter (q, seg, c2, c3)).  Both blocks are drawn even for a group of
// four or fewer at a segment's end (its extra normals are not stored): two
// independent Philox and Box-Muller chains without a branch between them
// interleave, 1.5-1.8 % faster on every workload measured.  Every normal --
// reference, benign noise, tamper direction -- takes the same accurate
// transform: a normal's error scales a live value's error by its
// coefficient, and near a cancellation a + c z ~ 0 the fp16 step is far
// below that coefficient.
__device__ __forceinline__ void normals8(const PhiloxRoundKeys &rk, uint32_t q0, uint32_t seg,
                                         uint32_t c2, uint32_t c3, float z[8]) {
  const float4 a = normals4_rk(rk, q0, seg, c2, c3);
  const float4 b = normals4_rk(rk, q0 + 1, seg, c2, c3);
  z[0] = a.x; z[1] = a.y; z[2] = a.z; z[3] = a.w;
  z[4] = b.x; z[5] = b.y; z[6] = b.z; z[7] = b.w;
}

// Bits 0..7 = mask bits of the channels c, c+1, ..., c+7 (wrapping at d).
// When 8 divides d, c (= e0 mod d with e0 a multiple of 8) is a multiple of
// 8, so the eight channels sit in one mask word and one load serves them.
__device__ __forceinline__ uint32_t channel_bits8(const uint32_t *mask, uint32_t c, uint32_t d) {
  if ((d & 7u) == 0) return (__ldg(mask + (c >> 5)) >> (c & 31u)) & 0xFFu;
  uint32_t bits = 0;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    bits |= (mask_bit(mask, c) ? 1u : 0u) << k;
    c = (c + 1 == d) ? 0 : c + 1;
  }
  return bits;
}

// Whether a stage's live values depend on statistics of the whole segment:
// benign under the Eq. 2 model (mu = ||a||_1 / (T d)), malicious under the
// Gaussian tamper (||v||, ||g||).  Every other segment's live values follow
// element by element from its references.
__device__ __forceinline__ bool needs_stats(const GenParams &p, bool mal) {
  return mal ? p.tamper == CG_TAMPER_ADDITIVE : p.noise == CG_NOISE_PAPER;
}

// fp16 live values of one group of 8, or in recompute mode their fp32
// copies written over the references.
__device__ __forceinline__ void store_live(const GenParams &p, uint16_t *acts, float *refs,
                                           uint64_t g, int cnt, bool vec, const float h[8]) {
  if (p.recompute) {
    if (vec) {
      float v[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) v[k] = __half2float(__float2half_rn(h[k]));
      float4 *r4 = reinterpret_cast<float4 *>(refs + g);
      r4[0] = make_float4(v[0], v[1], v[2], v[3]);
      r4[1] = make_float4(v[4], v[5], v[6], v[7]);
    } else {
      for (int k = 0; k < cnt; ++k) refs[g + k] = __half2float(__float2half_rn(h[k]));
    }
    return;
  }
  if (vec) {
    uint4 hv;
    hv.x = (uint32_t)__half_as_ushort(__float2half_rn(h[0])) |
           ((uint32_t)__half_as_ushort(__float2half_rn(h[1])) << 16);
    hv.y = (uint32_t)__half_as_ushort(__float2half_rn(h[2])) |
           ((uint32_t)__half_as_ushort(__float2half_rn(h[3])) << 16);
    hv.z = (uint32_t)__half_as_ushort(__float2half_rn(h[4])) |
           ((uint32_t)__half_as_ushort(__float2half_rn(h[5])) << 16);
    hv.w = (uint32_t)__half_as_ushort(__float2half_rn(h[6])) |
           ((uint32_t)__half_as_ushort(__float2half_rn(h[7])) << 16);
    *reinterpret_cast<uint4 *>(acts + g) = hv;
  } else {
    for (int k = 0; k < cnt; ++k) acts[g + k] = __half_as_ushort(__float2half_rn(h[k]));
  }
}

// ----------------------------------------------------------------- pass 1: references
// Work item = (segment, chunk of kGenStatChunk elements).  Each thread takes
// groups of 8 elements: two Philox blocks of reference normals, the
// reference a (outlier channels scaled), a 16-byte store pair when the
// group is whole and 8-aligned.
// kLive: on a segment whose live values need no segment statistics (benign
// a (1 + sigma_s z); sign flips; rescale) the live values are formed here
// from the registers and stored beside the references, and pass 2 skips
// the segment.  On the other segments the block reduces what their live
// values need: sum |a| on a benign stage under the Eq. 2 model, sum a^2 and
// the tamper direction's sum g^2 on a Gaussian-tamper stage.  One double2
// per item.  Without kLive only the references are written.
template <bool kLive>
__global__ void __launch_bounds__(kGenThreads)
gen_refs_kernel(GenParams p, const uint32_t *__restrict__ outlier_mask,
                const uint32_t *__restrict__ flip_mask, const float *__restrict__ stage_sigma,
                float *__restrict__ refs, uint16_t *__restrict__ acts,
                double2 *__restrict__ stats) {
  __shared__ double2 warp_sum[kGenThreads / 32];
  const uint64_t n_items = (uint64_t)p.S * p.N * p.stat_chunks;
  const PhiloxRoundKeys &rk = *reinterpret_cast<const PhiloxRoundKeys *>(p.round_keys);
  const uint32_t c2_ref = 4u * p.config_id + kStreamRef;
  const uint32_t c2_noise = 4u * p.config_id + kStreamNoise;
  const uint32_t c2_tamper = 4u * p.config_id + kStreamTamper;
  const uint32_t c_step = (uint32_t)((8ull * kGenThreads) % p.d);
  const int tid = threadIdx.x;
  for (uint64_t item = blockIdx.x; item < n_items; item += gridDim.x) {
    const uint32_t seg = (uint32_t)(item / p.stat_chunks);
    const uint64_t ch = item - (uint64_t)seg * p.stat_chunks;
    const uint32_t s = seg / p.N;
    const bool mal = is_malicious(p, s);
    const bool stat_seg = kLive && needs_stats(p, mal);
    const bool fused = kLive && !stat_seg;
    const bool need_l1 = stat_seg && !mal;
    const bool need_l2 = stat_seg && mal;
    const bool flips = fused && mal && p.tamper == CG_TAMPER_SIGNFLIP_CHANNELS;
    // the per-segment scalar of a fused segment: sigma_s (benign) or beta (rescale)
    const float cf = !fused ? 0.f : (mal ? p.tamper_param : stage_sigma[s]);
    const uint32_t *flip_row = flip_mask + (uint64_t)s * p.mask_words;
    const uint64_t seg_base = (uint64_t)seg * p.L;
    const uint64_t e_begin = ch * kGenStatChunk;
    const uint64_t e_end = min(e_begin + (uint64_t)kGenStatChunk, p.L);
    uint64_t e0 = e_begin + 8 * (uint64_t)tid;
    uint32_t c = (uint32_t)(e0 % p.d);                   // channel of element e0
    float x = 0.f, y = 0.f;
    for (; e0 < e_end; e0 += 8 * (uint64_t)kGenThreads) {
      const int cnt = (int)min((uint64_t)8, p.L - e0);
      const uint32_t q0 = (uint32_t)(e0 >> 2);
      float z[8], a[8];
      normals8(rk, q0, seg, c2_ref, 0u, z);
      const uint32_t obits = p.n_outlier > 0 ? channel_bits8(outlier_mask, c, p.d) : 0u;
#pragma unroll
      for (int k = 0; k < 8; ++k) a[k] = ((obits >> k) & 1u) ? z[k] * p.outlier_scale : z[k];
      const uint64_t gidx = seg_base + e0;
      const bool vec = cnt == 8 && (gidx & 7) == 0;
      if (need_l1) {
        for (int k = 0; k < cnt; ++k) x += fabsf(a[k]);
      } else if (need_l2) {
        float g[8];
        normals8(rk, q0, seg, c2_tamper, 0u, g);
        for (int k = 0; k < cnt; ++k) {
          x = fmaf(a[k], a[k], x);
          y = fmaf(g[k], g[k], y);
        }
      }
      if (fused) {
        float h[8];
        if (!mal) {
          float n[8];
          normals8(rk, q0, seg, c2_noise, p.noise_c3, n);
#pragma unroll
          for (int k = 0; k < 8; ++k) h[k] = a[k] * (1.0f + cf * n[k]);   // a (1 + sigma_s z)
        } else if (flips) {
          const uint32_t fbits = channel_bits8(flip_row, c, p.d);
#pragma unroll
          for (int k = 0; k < 8; ++k) h[k] = ((fbits >> k) & 1u) ? -a[k] : a[k];
        } else if (p.tamper == CG_TAMPER_SIGNFLIP_FULL) {
#pragma unroll
          for (int k = 0; k < 8; ++k) h[k] = -a[k];
        } else {
#pragma unroll
          for (int k = 0; k < 8; ++k) h[k] = cf * a[k];                    // beta a
        }
        store_live(p, acts, refs, gidx, cnt, vec, h);
        if (p.recompute) {
          c += c_step;
          if (c >= p.d) c -= p.d;
          continue;                                   // the recompute replaces the references
        }
      }
      if (vec) {
        float4 *r4 = reinterpret_cast<float4 *>(refs + gidx);
        r4[0] = make_float4(a[0], a[1], a[2], a[3]);
        r4[1] = make_float4(a[4], a[5], a[6], a[7]);
      } else {
        for (int k = 0; k < cnt; ++k) refs[gidx + k] = a[k];
      }
      c += c_step;
      if (c >= p.d) c -= p.d;
    }
    if (!stat_seg) continue;                         // uniform over the block
    double dx = x, dy = y;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      dx += __shfl_down_sync(0xFFFFFFFFu, dx, off);
      dy += __shfl_down_sync(0xFFFFFFFFu, dy, off);
    }
    if ((tid & 31) == 0) warp_sum[tid >> 5] = make_double2(dx, dy);
    __syncthreads();
    if (tid == 0) {
      double2 t = make_double2(0.0, 0.0);
      for (int w = 0; w < kGenThreads / 32; ++w) {
        t.x += warp_sum[w].x;
        t.y += warp_sum[w].y;
      }
      stats[item] = t;
    }
    __syncthreads();
  }
}

// ----------------------------------------------------------------- coef
// Per segment of stages s_first .. s_first + n_stages - 1: benign PAPER ->
// sigma_s * mu with mu = sum|a| / L (Eq. 2); malicious ADDITIVE ->
// eps sqrt(sum a^2 / sum g^2) (tau(v) = v + eps ||v|| g / ||g||); benign
// MULT -> sigma_s; SCALE -> beta; otherwise 0.  stat_only: only the
// segments whose live values need statistics (the others were finished in
// pass 1 and have no sums).  Fixed order, fp64.
__global__ void gen_coef_kernel(GenParams p, uint32_t s_first, uint32_t n_stages, int stat_only,
                                const double2 *__restrict__ stats,
                                const float *__restrict__ stage_sigma, float *__restrict__ coef) {
  const uint64_t seg = (uint64_t)s_first * p.N + (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (seg >= (uint64_t)(s_first + n_stages) * p.N) return;
  const uint32_t s = (uint32_t)(seg / p.N);
  if (stat_only && !needs_stats(p, is_malicious(p, s))) return;
  double x = 0.0, y = 0.0;
  const double2 *st = stats + seg * p.stat_chunks;
  for (uint64_t c = 0; c < p.stat_chunks; ++c) {
    x += st[c].x;
    y += st[c].y;
  }
  float v = 0.f;
  if (!is_malicious(p, s)) {
    v = (p.noise == CG_NOISE_PAPER) ? (float)((double)stage_sigma[s] * (x / (double)p.L))
                                    : stage_sigma[s];
  } else if (p.tamper == CG_TAMPER_ADDITIVE) {
    v = (y > 0.0) ? (float)((double)p.tamper_param * sqrt(x) / sqrt(y)) : 0.f;
  } else if (p.tamper == CG_TAMPER_SCALE) {
    v = p.tamper_param;
  }
  coef[seg] = v;
}

// ----------------------------------------------------------------- pass 2: live values
// The segments pass 1 left: benign under the Eq. 2 model (h = a + sigma_s mu
// z) and malicious under the Gaussian tamper (h = a + coef g), both
// h = fp16(a + coef w) with w the noise or tamper normal.  Work item =
// (segment, chunk of kLiveChunk elements); each thread takes groups of 8:
// the references read back (16-byte loads when the group is whole and
// 8-aligned), the normals drawn, the fp16 live values stored.  In recompute
// mode every stage is benign, its noise comes from counter word 3 = the
// replica, and the fp16 result overwrites the references in place as fp32.
constexpr uint64_t kLiveChunk = 8 * kGenThreads * 8;

__global__ void __launch_bounds__(kGenThreads)
gen_live_kernel(GenParams p, const float *__restrict__ coef, uint16_t *__restrict__ acts,
                float *__restrict__ refs) {
  const uint64_t chunks = (p.L + kLiveChunk - 1) / kLiveChunk;
  const uint64_t n_items = (uint64_t)p.S * p.N * chunks;
  const PhiloxRoundKeys &rk = *reinterpret_cast<const PhiloxRoundKeys *>(p.round_keys);
  const uint32_t c2_noise = 4u * p.config_id + kStreamNoise;
  const uint32_t c2_tamper = 4u * p.config_id + kStreamTamper;
  for (uint64_t item = blockIdx.x; item < n_items; item += gridDim.x) {
    const uint32_t seg = (uint32_t)(item / chunks);
    const uint32_t s = seg / p.N;
    const bool mal = is_malicious(p, s);
    if (!needs_stats(p, mal)) continue;
    const uint64_t ch = item - (uint64_t)seg * chunks;
    const float cf = coef[seg];
    const uint32_t c2 = mal ? c2_tamper : c2_noise;
    const uint32_t c3 = mal ? 0u : p.noise_c3;
    const uint64_t seg_base = (uint64_t)seg * p.L;
    const uint64_t e_end = min((ch + 1) * kLiveChunk, p.L);
    for (uint64_t e0 = ch * kLiveChunk + 8 * (uint64_t)threadIdx.x; e0 < e_end;
         e0 += 8 * (uint64_t)kGenThreads) {
      const int cnt = (int)min((uint64_t)8, p.L - e0);
      const uint64_t g = seg_base + e0;
      const bool vec = cnt == 8 && (g & 7) == 0;
      float a[8], w[8], h[8];
      if (vec) {
        const float4 r0 = reinterpret_cast<const float4 *>(refs + g)[0];
        const float4 r1 = reinterpret_cast<const float4 *>(refs + g)[1];
        a[0] = r0.x; a[1] = r0.y; a[2] = r0.z; a[3] = r0.w;
        a[4] = r1.x; a[5] = r1.y; a[6] = r1.z; a[7] = r1.w;
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) a[k] = (k < cnt) ? refs[g + k] : 0.f;
      }
      normals8(rk, (uint32_t)(e0 >> 2), seg, c2, c3, w);
#pragma unroll
      for (int k = 0; k < 8; ++k) h[k] = fmaf(cf, w[k], a[k]);           // a + coef w
      store_live(p, acts, refs, g, cnt, vec, h);
    }
  }
}

// ----------------------------------------------------------------- propagating pipeline
// Eq. 2's recursion with the block's response to its input linearised:
//   v_s = f_s(h_{s-1}) = a_s + gain (h_{s-1} - a_{s-1}),  v_0 = a_0,
// benign h_s = fp16(v_s + sigma_s mu_s z) (mu_s = ||v_s||_1 / (T d)) or
// fp16(v_s (1 + sigma_s z)); malicious h_s = fp16(tau(v_s)).  Stage s reads
// stage s-1's stored fp16 live values and fp32 references, so the stages
// run one after the other.
__device__ __forceinline__ void prop_inputs(const GenParams &p, uint32_t s, float gain,
                                            const float *refs, const uint16_t *acts, uint64_t g,
                                            uint64_t gprev, int cnt, bool vec, float v[8]) {
  float a[8], ap[8], hp[8];
  if (vec) {
    const float4 r0 = reinterpret_cast<const float4 *>(refs + g)[0];
    const float4 r1 = reinterpret_cast<const float4 *>(refs + g)[1];
    a[0] = r0.x; a[1] = r0.y; a[2] = r0.z; a[3] = r0.w;
    a[4] = r1.x; a[5] = r1.y; a[6] = r1.z; a[7] = r1.w;
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) a[k] = (k < cnt) ? refs[g + k] : 0.f;
  }
  if (s == 0) {
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = a[k];
    return;
  }
  if (vec) {
    const float4 r0 = reinterpret_cast<const float4 *>(refs + gprev)[0];
    const float4 r1 = reinterpret_cast<const float4 *>(refs + gprev)[1];
    ap[0] = r0.x; ap[1] = r0.y; ap[2] = r0.z; ap[3] = r0.w;
    ap[4] = r1.x; ap[5] = r1.y; ap[6] = r1.z; ap[7] = r1.w;
    const uint4 hv = *reinterpret_cast<const uint4 *>(acts + gprev);
    const uint32_t w[4] = {hv.x, hv.y, hv.z, hv.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      hp[2 * k] = __half2float(__ushort_as_half((uint16_t)(w[k] & 0xFFFFu)));
      hp[2 * k + 1] = __half2float(__ushort_as_half((uint16_t)(w[k] >> 16)));
    }
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      ap[k] = (k < cnt) ? refs[gprev + k] : 0.f;
      hp[k] = (k < cnt) ? __half2float(__ushort_as_half(acts[gprev + k])) : 0.f;
    }
  }
#pragma unroll
  for (int k = 0; k < 8; ++k) v[k] = fmaf(gain, hp[k] - ap[k], a[k]);
}

__global__ void __launch_bounds__(kGenThreads)
gen_prop_stats_kernel(GenParams p, uint32_t s, float gain, const float *__restrict__ refs,
                      const uint16_t *__restrict__ acts, double2 *__restrict__ stats) {
  __shared__ double2 warp_sum[kGenThreads / 32];
  const uint64_t n_items = (uint64_t)p.N * p.stat_chunks;
  const PhiloxRoundKeys &rk = *reinterpret_cast<const PhiloxRoundKeys *>(p.round_keys);
  const uint32_t c2_tamper = 4u * p.config_id + kStreamTamper;
  const bool mal = is_malicious(p, s);
  const bool need_l1 = !mal && p.noise == CG_NOISE_PAPER;
  const bool need_l2 = mal && p.tamper == CG_TAMPER_ADDITIVE;
  const int tid = threadIdx.x;
  for (uint64_t it = blockIdx.x; it < n_items; it += gridDim.x) {
    const uint32_t n = (uint32_t)(it / p.stat_chunks);
    const uint64_t ch = it - (uint64_t)n * p.stat_chunks;
    const uint32_t seg = s * p.N + n;
    const uint64_t e_begin = ch * kGenStatChunk;
    const uint64_t e_end = min(e_begin + (uint64_t)kGenStatChunk, p.L);
    float x = 0.f, y = 0.f;
    if (need_l1 || need_l2) {
      for (uint64_t e0 = e_begin + 8 * (uint64_t)tid; e0 < e_end;
           e0 += 8 * (uint64_t)kGenThreads) {
        const int cnt = (int)min((uint64_t)8, p.L - e0);
        const uint64_t g = (uint64_t)seg * p.L + e0;
        const uint64_t gprev = g - (s ? (uint64_t)p.N * p.L : 0);
        const bool vec = (cnt == 8) && ((g & 7) == 0) && ((gprev & 7) == 0);
        float v[8];
        prop_inputs(p, s, gain, refs, acts, g, gprev, cnt, vec, v);
        if (need_l1) {
          for (int k = 0; k < cnt; ++k) x += fabsf(v[k]);
        } else {
          float gg[8];
          normals8(rk, (uint32_t)(e0 >> 2), seg, c2_tamper, 0u, gg);
          for (int k = 0; k < cnt; ++k) {
            x = fmaf(v[k], v[k], x);
            y = fmaf(gg[k], gg[k], y);
          }
        }
      }
    }
    double dx = x, dy = y;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      dx += __shfl_down_sync(0xFFFFFFFFu, dx, off);
      dy += __shfl_down_sync(0xFFFFFFFFu, dy, off);
    }
    if ((tid & 31) == 0) warp_sum[tid >> 5] = make_double2(dx, dy);
    __syncthreads();
    if (tid == 0) {
      double2 t = make_double2(0.0, 0.0);
      for (int w = 0; w < kGenThreads / 32; ++w) {
        t.x += warp_sum[w].x;
        t.y += warp_sum[w].y;
      }
      stats[(uint64_t)seg * p.stat_chunks + ch] = t;
    }
    __syncthreads();
  }
}

__global__ void __launch_bounds__(kGenThreads)
gen_prop_live_kernel(GenParams p, uint32_t s, float gain, const uint32_t *__restrict__ flip_mask,
                     const float *__restrict__ coef, const float *__restrict__ refs,
                     uint16_t *__restrict__ acts) {
  const uint64_t groups_per_seg = (p.L + 7) >> 3;
  const uint64_t total = (uint64_t)p.N * groups_per_seg;
  const PhiloxRoundKeys &rk = *reinterpret_cast<const PhiloxRoundKeys *>(p.round_keys);
  const uint32_t c2_noise = 4u * p.config_id + kStreamNoise;
  const uint32_t c2_tamper = 4u * p.config_id + kStreamTamper;
  const bool mal = is_malicious(p, s);
  for (uint64_t gi = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; gi < total;
       gi += (uint64_t)gridDim.x * blockDim.x) {
    const uint32_t n = (uint32_t)(gi / groups_per_seg);
    const uint64_t j = gi - (uint64_t)n * groups_per_seg;
    const uint32_t seg = s * p.N + n;
    const uint64_t e0 = 8 * j;
    const int cnt = (int)min((uint64_t)8, p.L - e0);
    const uint32_t q0 = (uint32_t)(2 * j);
    const uint64_t g = (uint64_t)seg * p.L + e0;
    const uint64_t gprev = g - (s ? (uint64_t)p.N * p.L : 0);
    const bool vec = (cnt == 8) && ((g & 7) == 0) && ((gprev & 7) == 0);
    float v[8], h[8];
    prop_inputs(p, s, gain, refs, acts, g, gprev, cnt, vec, v);
    const float cf = coef[seg];
    if (!mal || p.tamper == CG_TAMPER_ADDITIVE) {
      float z[8];
      normals8(rk, q0, seg, mal ? c2_tamper : c2_noise, 0u, z);
      if (!mal && p.noise == CG_NOISE_MULT) {
#pragma unroll
        for (int k = 0; k < 8; ++k) h[k] = v[k] * (1.0f + cf * z[k]);
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) h[k] = fmaf(cf, z[k], v[k]);
      }
    } else if (p.tamper == CG_TAMPER_SIGNFLIP_CHANNELS) {
      const uint32_t fbits =
          channel_bits8(flip_mask + (uint64_t)s * p.mask_words, (uint32_t)(e0 % p.d), p.d);
#pragma unroll
      for (int k = 0; k < 8; ++k) h[k] = ((fbits >> k) & 1u) ? -v[k] : v[k];
    } else if (p.tamper == CG_TAMPER_SIGNFLIP_FULL) {
#pragma unroll
      for (int k = 0; k < 8; ++k) h[k] = -v[k];
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) h[k] = cf * v[k];
    }
    if (vec) {
      uint4 hv;
      hv.x = (uint32_t)__half_as_ushort(__float2half_rn(h[0])) |
             ((uint32_t)__half_as_ushort(__float2half_rn(h[1])) << 16);
      hv.y = (uint32_t)__half_as_ushort(__float2half_rn(h[2])) |
             ((uint32_t)__half_as_ushort(__float2half_rn(h[3])) << 16);
      hv.z = (uint32_t)__half_as_ushort(__float2half_rn(h[4])) |
             ((uint32_t)__half_as_ushort(__float2half_rn(h[5])) << 16);
      hv.w = (uint32_t)__half_as_ushort(__float2half_rn(h[6])) |
             ((uint32_t)__half_as_ushort(__float2half_rn(h[7])) << 16);
      *reinterpret_cast<uint4 *>(acts + g) = hv;
    } else {
      for (int k = 0; k < cnt; ++k) acts[g + k] = __half_as_ushort(__float2half_rn(h[k]));
    }
  }
}

// ----------------------------------------------------------------- random baseline
// Sec. 4.5: every score replaced by Uniform(0, 1).  Score (c, n, s) is
// (x >> 8) 2^-24 with x word s of aux stream (RANDOM, canary n) of config id
// config_id0 + c, i.e. word s % 4 of the Philox block with counter
// (s / 4, RANDOM << 24 | n, 4 (config_id0 + c) + 3, 0).  A thread makes one
// such block: four consecutive scores of one row, one 16-byte store when the
// row's four scores are 16-byte aligned, so a warp writes 512 contiguous
// bytes.  Grid-stride over the C N ceil(S / 4) blocks.  Below 2^32 blocks
// the index splits take 32-bit division by multiplication with a
// precomputed reciprocal: for 32-bit n and d >= 2, n / d is the high 64 bits
// of n ceil(2^64 / d) (Lemire, Kaser and Kurz, "Faster remainder by direct
// computation", 2019).  The round keys come precomputed, as in the generator.
__device__ __forceinline__ uint32_t div_by_recip(uint32_t n, uint64_t recip, uint32_t d) {
  return d == 1 ? n : (uint32_t)__umul64hi(recip, (uint64_t)n);
}

constexpr int kRandomBlocksPerSm = 16;

template <bool kIdx32>
__global__ void __launch_bounds__(256)
random_scores_kernel(PhiloxRoundKeys rk, uint32_t config_id0, uint32_t N, uint32_t S,
                     uint64_t total, uint64_t recip_row, uint64_t recip_n,
                     float *__restrict__ out) {
  const uint32_t per_row = (S + 3u) / 4u;
  for (uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (uint64_t)gridDim.x * blockDim.x) {
    uint64_t row;
    uint32_t q, c, n;
    if (kIdx32) {
      const uint32_t t32 = (uint32_t)t;
      const uint32_t r32 = div_by_recip(t32, recip_row, per_row);
      q = t32 - r32 * per_row;
      c = div_by_recip(r32, recip_n, N);
      n = r32 - c * N;
      row = r32;
    } else {
      row = t / per_row;
      q = (uint32_t)(t - row * per_row);
      c = (uint32_t)(row / N);
      n = (uint32_t)(row - (uint64_t)c * N);
    }
    const uint4 w = philox4x32_10_rk(
        make_uint4(q, (kAuxRandom << 24) | (n & 0x00FFFFFFu), 4u * (config_id0 + c) + kStreamAux, 0u),
        rk);
    const float v0 = (float)(w.x >> 8) * 0x1p-24f, v1 = (float)(w.y >> 8) * 0x1p-24f;
    const float v2 = (float)(w.z >> 8) * 0x1p-24f, v3 = (float)(w.w >> 8) * 0x1p-24f;
    float *o = out + row * S + 4ull * q;
    if ((S & 3u) == 0 && ((uintptr_t)o & 15u) == 0) {
      *reinterpret_cast<float4 *>(o) = make_float4(v0, v1, v2, v3);
    } else {
      const uint32_t m = min(4u, S - 4u * q);
      o[0] = v0;
      if (m > 1) o[1] = v1;
      if (m > 2) o[2] = v2;
      if (m > 3) o[3] = v3;
    }
  }
}

// ----------------------------------------------------------------- test views
__global__ void philox_words_kernel(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                                    uint32_t first, uint32_t n, uint4 *out) {
  const uint32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  out[i] = philox4x32_10(make_uint4(first + i, c1, c2, c3), philox_key(seed));
}

__global__ void philox_normals_kernel(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                                      uint32_t first, uint32_t n, float4 *out) {
  const uint32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint4 w = philox4x32_10(make_uint4(first + i, c1, c2, c3), philox_key(seed));
  const float2 a = box_muller(w.x, w.y), b = box_muller(w.z, w.w);
  out[i] = make_float4(a.x, a.y, b.x, b.y);
}

__global__ void box_muller_pairs_kernel(const uint2 *__restrict__ words, uint64_t n,
                                        float2 *__restrict__ out) {
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (uint64_t)gridDim.x * blockDim.x) {
    const uint2 w = words[i];
    out[i] = box_muller(w.x, w.y);
  }
}

// Whether any segment's live values need segment statistics (pass 2).
bool host_any_stats(const GenParams &p) {
  bool any_mal = false, any_benign = false;
  for (uint32_t s = 0; s < p.S; ++s) {
    if ((p.mal_bits[s >> 5] >> (s & 31)) & 1u) any_mal = true;
    else any_benign = true;
  }
  return (any_benign && p.noise == CG_NOISE_PAPER) || (any_mal && p.tamper == CG_TAMPER_ADDITIVE);
}

}  // namespace

GenLayout gen_layout(const cg_pipeline_desc &d) {
  GenLayout g;
  const uint64_t L = (uint64_t)d.tokens * d.hidden;
  g.mask_words = (d.hidden + 31) / 32;
  g.stat_chunks = (L + kGenStatChunk - 1) / kGenStatChunk;
  const uint64_t n_seg = (uint64_t)d.n_shards * d.n_canaries;
  size_t off = 256;   // reserved
  g.outlier_mask = off;
  off = align_up(off + (size_t)g.mask_words * 4, 256);
  g.flip_mask = off;
  off = align_up(off + (size_t)d.n_shards * g.mask_words * 4, 256);
  g.stage_sigma = off;
  off = align_up(off + (size_t)d.n_shards * 4, 256);
  g.seg_coef = off;
  off = align_up(off + (size_t)n_seg * 4, 256);
  g.stats = off;
  off = align_up(off + (size_t)(n_seg * g.stat_chunks) * 16, 256);
  g.total = off;
  return g;
}

cudaError_t launch_generate(const GenParams &p, uint16_t *acts, float *refs, int8_t *labels,
                            void *ws, const GenLayout &lay, int32_t *status, cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  char *base = static_cast<char *>(ws);
  uint32_t *outlier_mask = reinterpret_cast<uint32_t *>(base + lay.outlier_mask);
  uint32_t *flip_mask = reinterpret_cast<uint32_t *>(base + lay.flip_mask);
  float *stage_sigma = reinterpret_cast<float *>(base + lay.stage_sigma);
  float *coef = reinterpret_cast<float *>(base + lay.seg_coef);
  double2 *stats = reinterpret_cast<double2 *>(base + lay.stats);

  cudaError_t err;
  gen_setup_kernel<<<1, 256, 0, stream>>>(p, outlier_mask, flip_mask, stage_sigma, labels, status);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;

  const uint64_t n_seg = (uint64_t)p.S * p.N;
  const uint64_t resident = (uint64_t)info.sm_count * (uint64_t)info.gen_blocks_per_sm;
  const uint64_t n_items = n_seg * p.stat_chunks;
  const uint64_t grid1 = n_items < resident ? n_items : resident;
  gen_refs_kernel<true><<<(unsigned)grid1, kGenThreads, 0, stream>>>(
      p, outlier_mask, flip_mask, stage_sigma, refs, acts, stats);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  if (!host_any_stats(p)) return cudaSuccess;       // pass 1 finished every segment

  gen_coef_kernel<<<(unsigned)((n_seg + 127) / 128), 128, 0, stream>>>(p, 0, p.S, 1, stats,
                                                                       stage_sigma, coef);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  const uint64_t live_items = n_seg * ((p.L + kLiveChunk - 1) / kLiveChunk);
  const uint64_t resident2 = (uint64_t)info.sm_count * (uint64_t)info.gen_live_blocks_per_sm;
  const uint64_t grid2 = live_items < resident2 ? live_items : resident2;
  gen_live_kernel<<<(unsigned)grid2, kGenThreads, 0, stream>>>(p, coef, acts, refs);
  return cudaGetLastError();
}

cudaError_t launch_generate_propagating(const GenParams &p, float gain, uint16_t *acts, float *refs,
                                       int8_t *labels, void *ws, const GenLayout &lay,
                                       int32_t *status, cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  char *base = static_cast<char *>(ws);
  uint32_t *outlier_mask = reinterpret_cast<uint32_t *>(base + lay.outlier_mask);
  uint32_t *flip_mask = reinterpret_cast<uint32_t *>(base + lay.flip_mask);
  float *stage_sigma = reinterpret_cast<float *>(base + lay.stage_sigma);
  float *coef = reinterpret_cast<float *>(base + lay.seg_coef);
  double2 *stats = reinterpret_cast<double2 *>(base + lay.stats);
  cudaError_t err;
  gen_setup_kernel<<<1, 256, 0, stream>>>(p, outlier_mask, flip_mask, stage_sigma, labels, status);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  const uint64_t n_seg = (uint64_t)p.S * p.N;
  const uint64_t resident = (uint64_t)info.sm_count * (uint64_t)info.gen_blocks_per_sm;
  // every stage's reference first (its statistics are recomputed below)
  const uint64_t n_items = n_seg * p.stat_chunks;
  gen_refs_kernel<false><<<(unsigned)(n_items < resident ? n_items : resident), kGenThreads, 0,
                          stream>>>(p, outlier_mask, flip_mask, stage_sigma, refs, nullptr, nullptr);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  const uint64_t stage_items = (uint64_t)p.N * p.stat_chunks;
  const uint64_t stage_groups = (uint64_t)p.N * ((p.L + 7) >> 3);
  const uint64_t live_blocks = (stage_groups + kGenThreads - 1) / kGenThreads;
  for (uint32_t s = 0; s < p.S; ++s) {
    gen_prop_stats_kernel<<<(unsigned)(stage_items < resident ? stage_items : resident), kGenThreads,
                            0, stream>>>(p, s, gain, refs, acts, stats);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    gen_coef_kernel<<<(unsigned)((p.N + 127) / 128), 128, 0, stream>>>(p, s, 1, 0, stats,
                                                                       stage_sigma, coef);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    gen_prop_live_kernel<<<(unsigned)(live_blocks < resident * 4 ? live_blocks : resident * 4),
                           kGenThreads, 0, stream>>>(p, s, gain, flip_mask, coef, refs, acts);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
  }
  return cudaSuccess;
}

cudaError_t launch_random_scores(uint64_t seed, uint32_t config_id0, uint32_t C, uint32_t N,
                                 uint32_t S, float *out, cudaStream_t stream) {
  const uint32_t per_row = (S + 3u) / 4u;
  const uint64_t total = (uint64_t)C * N * per_row;
  PhiloxRoundKeys rk;
  uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  for (int r = 0; r < 10; ++r) {
    rk.k[2 * r] = k0;
    rk.k[2 * r + 1] = k1;
    k0 += kPhiloxW0;
    k1 += kPhiloxW1;
  }
  // ceil(2^64 / d) for d >= 2 (unused for d = 1)
  auto recip = [](uint32_t d) -> uint64_t { return d < 2 ? 0 : UINT64_MAX / d + 1; };
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  const uint64_t blocks = (total + 255) / 256;
  const uint64_t cap = (uint64_t)info.sm_count * kRandomBlocksPerSm;   // grid-stride beyond
  const unsigned grid = (unsigned)(blocks < cap ? blocks : cap);
  if (total < (1ull << 32)) {
    random_scores_kernel<true><<<grid, 256, 0, stream>>>(rk, config_id0, N, S, total,
                                                        recip(per_row), recip(N), out);
  } else {
    random_scores_kernel<false><<<grid, 256, 0, stream>>>(rk, config_id0, N, S, total, 0, 0, out);
  }
  return cudaGetLastError();
}

cudaError_t launch_philox_words(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                                uint32_t first, uint32_t n, uint32_t *out, cudaStream_t stream) {
  philox_words_kernel<<<(n + 255) / 256, 256, 0, stream>>>(seed, c1, c2, c3, first, n,
                                                           reinterpret_cast<uint4 *>(out));
  return cudaGetLastError();
}

cudaError_t launch_philox_normals(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                                  uint32_t first, uint32_t n, float *out, cudaStream_t stream) {
  philox_normals_kernel<<<(n + 255) / 256, 256, 0, stream>>>(seed, c1, c2, c3, first, n,
                                                             reinterpret_cast<float4 *>(out));
  return cudaGetLastError();
}

cudaError_t launch_box_muller_pairs(const uint32_t *words, uint64_t n_pairs, float *out,
                                   cudaStream_t stream) {
  const uint64_t blocks = (n_pairs + 255) / 256;
  box_muller_pairs_kernel<<<(unsigned)(blocks < 65536 ? blocks : 65536), 256, 0, stream>>>(
      reinterpret_cast<const uint2 *>(words), n_pairs, reinterpret_cast<float2 *>(out));
  return cudaGetLastError();
}

// Generator blocks per SM: the occupancy of pass 1, capped at kGenBlocksPerSm
// so that one drift block (288 threads x 32 registers, 147 KB of shared
// memory) still fits beside them.  A caller that scores one configuration
// while it generates the next on another stream then overlaps the two: the
// generator is bound by integer/FP32 issue, the drift reduction by HBM.  At
// 4 blocks per SM instead of 3 pass 1 is about 1 % faster alone and the
// studies 0.2-1.4 % faster, too little to give up that room.
int gen_occupancy() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gen_refs_kernel<true>, kGenThreads, 0) !=
      cudaSuccess)
    return 0;
  return n < kGenBlocksPerSm ? n : kGenBlocksPerSm;
}

// Blocks per SM of pass 2 (gen_live_kernel): all its registers allow (6 of
// 256 threads at 40 registers), not capped like pass 1.  Pass 2 is bound by
// integer/FP32 issue too, and more resident warps hide more of its latency:
// 70B-like generator 14.95 -> 14.58 ms, factorial study 1,419 -> 1,449
// configs/s although a co-running drift block then waits for room on the SM.
int gen_live_occupancy() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gen_live_kernel, kGenThreads, 0) !=
      cudaSuccess)
    return 0;
  return n;
}

}  // namespace cg
