// drift.cu -- the per-(stage, canary) drift reduction (Eq. 4 and the cosine
// mismatch of the Sec. 4.4 ablation), the HBM-bound hot loop of the
// verifier: every fp16 live element and every fp32 reference element is
// read exactly once (6 bytes per element).
//
// Pass 1 cuts the [C][S][N][L] element space into work items of at most
// kDriftChunk elements (drift_item_len: even shares of a segment in whole
// 4,096-element stages), never crossing a segment, and writes one float4 of
// fp32 sums per item:
//     D = sum (h - a)^2,   E = sum (h - a)(h + a) = sum h^2 - a^2,
//     A = sum a^2,         M = max |h - a|
// by one of two kernels:
//   drift_bulk_kernel     (default for device memory, seg_len % 8 == 0) a TMA
//                         pipeline: one producer warp fills a shared-memory
//                         ring with cp.async.bulk copies tracked by mbarriers,
//                         eight consumer warps accumulate;
//   drift_partial_kernel  (any seg_len, host-resident input, the no-alloc
//                         entry point) a persistent grid whose threads keep
//                         four 16-byte vectors per stream in flight with
//                         non-allocating, 256-byte-prefetching loads.
// Pass 2 (drift_finalize_kernel) combines the items of a segment in a fixed
// order in fp64 and writes the three scores.  No atomics, so the result is
// the same on every run.
#include <cuda_fp16.h>

#include <mutex>

#include "cg_internal.h"

namespace cg {
namespace {

struct Acc {
  float d, e, a, m;
};

__device__ __forceinline__ void acc_one(float h, float a, Acc &s) {
  const float diff = h - a;
  s.d = fmaf(diff, diff, s.d);
  s.e = fmaf(diff, h + a, s.e);
  s.a = fmaf(a, a, s.a);
  s.m = fmaxf(s.m, fabsf(diff));
}

__device__ __forceinline__ uint4 ld_stream(const void *p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

__device__ __forceinline__ float2 half2_bits_to_float2(uint32_t bits) {
  __half2 h;
  memcpy(&h, &bits, 4);
  return __half22float2(h);
}

// Eight elements: hv = 8 halves, r0/r1 = 8 floats.  A local sum of the
// eight terms is added to the running sums (shorter fp32 chains).
__device__ __forceinline__ void acc_eight(const uint4 hv, const uint4 r0, const uint4 r1, Acc &s) {
  Acc t = {0.f, 0.f, 0.f, s.m};
  float2 h;
  h = half2_bits_to_float2(hv.x);
  acc_one(h.x, __uint_as_float(r0.x), t);
  acc_one(h.y, __uint_as_float(r0.y), t);
  h = half2_bits_to_float2(hv.y);
  acc_one(h.x, __uint_as_float(r0.z), t);
  acc_one(h.y, __uint_as_float(r0.w), t);
  h = half2_bits_to_float2(hv.z);
  acc_one(h.x, __uint_as_float(r1.x), t);
  acc_one(h.y, __uint_as_float(r1.y), t);
  h = half2_bits_to_float2(hv.w);
  acc_one(h.x, __uint_as_float(r1.z), t);
  acc_one(h.y, __uint_as_float(r1.w), t);
  s.d += t.d;
  s.e += t.e;
  s.a += t.a;
  s.m = t.m;
}

__device__ __forceinline__ float half_bits_to_float(uint16_t b) {
  return __half2float(__ushort_as_half(b));
}

constexpr int kUnroll = 4;

__global__ void __launch_bounds__(kDriftThreads)
drift_partial_kernel(const uint16_t *__restrict__ acts, const float *__restrict__ refs,
                     uint64_t L, uint64_t chunks_per_seg, uint64_t item_len, uint64_t n_items,
                     float4 *__restrict__ partials) {
  __shared__ Acc warp_acc[kDriftThreads / 32];
  const int tid = threadIdx.x;
  for (uint64_t item = blockIdx.x; item < n_items; item += gridDim.x) {
    const uint64_t seg = item / chunks_per_seg;
    const uint64_t ch = item - seg * chunks_per_seg;
    const uint64_t seg0 = seg * L;
    const uint64_t g0 = seg0 + ch * item_len;
    const uint64_t g1 = min(g0 + item_len, seg0 + L);
    Acc s = {0.f, 0.f, 0.f, 0.f};

    uint64_t v0 = (g0 + 7) & ~(uint64_t)7;
    uint64_t v1 = g1 & ~(uint64_t)7;
    if (v0 >= v1) {          // no aligned 8-vector inside: all scalar
      v0 = g1;
      v1 = g1;
    }
    // scalar head [g0, v0) and tail [v1, g1): fewer than 8 elements each,
    // or the whole item when it has no aligned vector
    for (uint64_t g = g0 + tid; g < v0; g += kDriftThreads)
      acc_one(half_bits_to_float(acts[g]), refs[g], s);
    for (uint64_t g = v1 + tid; g < g1; g += kDriftThreads)
      acc_one(half_bits_to_float(acts[g]), refs[g], s);

    const uint64_t nv = (v1 - v0) >> 3;
    for (uint64_t i = tid; i < nv; i += (uint64_t)kUnroll * kDriftThreads) {
      uint4 hv[kUnroll], r0[kUnroll], r1[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const uint64_t k = i + (uint64_t)u * kDriftThreads;
        if (k < nv) {
          const uint64_t g = v0 + 8 * k;
          hv[u] = ld_stream(acts + g);
          r0[u] = ld_stream(refs + g);
          r1[u] = ld_stream(refs + g + 4);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if (i + (uint64_t)u * kDriftThreads < nv) acc_eight(hv[u], r0[u], r1[u], s);
      }
    }

    // block reduction: shuffle tree inside each warp, then warp 0 in order
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      s.d += __shfl_down_sync(0xFFFFFFFFu, s.d, off);
      s.e += __shfl_down_sync(0xFFFFFFFFu, s.e, off);
      s.a += __shfl_down_sync(0xFFFFFFFFu, s.a, off);
      s.m = fmaxf(s.m, __shfl_down_sync(0xFFFFFFFFu, s.m, off));
    }
    if ((tid & 31) == 0) warp_acc[tid >> 5] = s;
    __syncthreads();
    if (tid < 32) {
      Acc t = (tid < kDriftThreads / 32) ? warp_acc[tid] : Acc{0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int off = 4; off > 0; off >>= 1) {
        t.d += __shfl_down_sync(0xFFFFFFFFu, t.d, off);
        t.e += __shfl_down_sync(0xFFFFFFFFu, t.e, off);
        t.a += __shfl_down_sync(0xFFFFFFFFu, t.a, off);
        t.m = fmaxf(t.m, __shfl_down_sync(0xFFFFFFFFu, t.m, off));
      }
      if (tid == 0) partials[item] = make_float4(t.d, t.e, t.a, t.m);
    }
    __syncthreads();   // warp_acc is reused by the next item
  }
}

// Scores of one segment from its fp64 sums.
//   rel_l2  = sqrt(D / A)                                  (Eq. 4)
//   cos_dev = 1 - h.a / (|h| |a|) with H = A + E, evaluated as
//             (D - E^2 / (sqrt H + sqrt A)^2) / (2 sqrt(H A)), which equals
//             (D - (sqrt H - sqrt A)^2) / (2 sqrt(H A)) without cancelling
//             two near-equal norms.
// G = 2^log_g lanes per segment (the smallest power of two that leaves each
// lane at most 8 items, at most 32): lane l of the group adds the items
// l, l + G, ... in order in fp64, then a fixed shuffle tree combines the
// group.  A segment of few items thus takes few lanes (3 items: one lane, so
// a warp finishes 32 segments), and a long one a whole warp.  Segment
// q = (c S + s) N + n of C configurations writes its scores at
// stat * stat_stride + c N S + n S + s.
constexpr int kFinThreads = 256;

__global__ void __launch_bounds__(kFinThreads)
drift_finalize_kernel(const float4 *__restrict__ partials, uint64_t chunks_per_seg, uint32_t C,
                      uint32_t S, uint32_t N, float *__restrict__ scores, uint64_t stat_stride,
                      int log_g) {
  const int G = 1 << log_g;
  const uint64_t seg = ((uint64_t)blockIdx.x * kFinThreads + threadIdx.x) >> log_g;
  const int sub = threadIdx.x & (G - 1);
  const uint64_t per_config = (uint64_t)S * N;
  const bool live = seg < (uint64_t)C * per_config;
  double D = 0.0, E = 0.0, A = 0.0;
  float M = 0.f;
  if (live) {
    const float4 *p = partials + seg * chunks_per_seg;
    for (uint64_t c = sub; c < chunks_per_seg; c += G) {
      const float4 v = p[c];
      D += (double)v.x;
      E += (double)v.y;
      A += (double)v.z;
      M = fmaxf(M, v.w);
    }
  }
  for (int off = G >> 1; off > 0; off >>= 1) {
    D += __shfl_down_sync(0xFFFFFFFFu, D, off, G);
    E += __shfl_down_sync(0xFFFFFFFFu, E, off, G);
    A += __shfl_down_sync(0xFFFFFFFFu, A, off, G);
    M = fmaxf(M, __shfl_down_sync(0xFFFFFFFFu, M, off, G));
  }
  if (!live || sub != 0) return;
  // The sums stay fp64; the scores are formed in fp32 from them (GB300's
  // FP64 pipe is narrow, and fp32 sqrt/div of the rounded sums is accurate
  // to a few 1e-7 relative, far inside the drift tolerances).
  float rel, cosd;
  // D >= M^2 holds for the exact sums, so D == 0 with M > 0 means every
  // squared difference underflowed fp32 (all |h - a| below about 2^-74.5):
  // the segment lies below the range the fp32 sums resolve, and its scores
  // are NaN rather than a wrong number.
  const bool underflow = (M > 0.f) && (D == 0.0);
  if (isnan(D) || isnan(A) || underflow) {
    rel = NAN;
  } else if (A > 0.0) {
    rel = sqrtf((float)D / (float)A);
  } else {
    rel = (D == 0.0) ? 0.f : INFINITY;
  }
  const double H = A + E;
  if (isnan(D) || isnan(E) || isnan(A) || underflow) {
    cosd = NAN;
  } else if (H > 0.0 && A > 0.0 && (isinf(D) || isinf(E))) {
    cosd = NAN;                                  // an infinite live element: h / |h| is inf / inf
  } else if (H > 0.0 && A > 0.0) {
    const float sh = sqrtf((float)H), sa = sqrtf((float)A);
    const float gap = (float)E / (sh + sa);
    cosd = ((float)D - gap * gap) / (2.0f * sh * sa);
    cosd = fminf(fmaxf(cosd, 0.f), 2.f);
  } else {
    cosd = 0.f;
  }
  const uint64_t c = seg / per_config, r = seg - c * per_config;
  const uint32_t s = (uint32_t)(r / N), n = (uint32_t)(r % N);
  const uint64_t o = c * per_config + (uint64_t)n * S + s;
  scores[o] = rel;
  scores[stat_stride + o] = M;
  scores[2 * stat_stride + o] = cosd;
}

static cudaError_t launch_finalize(const float4 *partials, uint64_t cps, uint32_t C, uint32_t S,
                                   uint32_t N, float *scores, uint64_t stat_stride,
                                   cudaStream_t stream) {
  const uint64_t n_seg = (uint64_t)C * S * N;
  int log_g = 0;                                   // lanes per segment: 2^log_g
  while (log_g < 5 && ((uint64_t)8 << log_g) < cps) ++log_g;
  const uint64_t blocks = ((n_seg << log_g) + kFinThreads - 1) / kFinThreads;
  drift_finalize_kernel<<<(unsigned)blocks, kFinThreads, 0, stream>>>(partials, cps, C, S, N,
                                                                      scores, stat_stride, log_g);
  return cudaGetLastError();
}

// ----------------------------------------------------------------- TMA bulk pipeline
// drift_bulk_kernel: the same work items and per-item float4 partials as
// drift_partial_kernel, but the bytes are staged through shared memory by
// the Tensor Memory Accelerator's 1-D bulk copies:
//   warp 0, lane 0   producer: for every stage (<= kBulkStageElems elements
//                    of one item) waits for its ring slot to be released,
//                    arms the slot's `full` mbarrier with the byte count and
//                    issues two cp.async.bulk copies (fp16 live, fp32 ref);
//                    at the start of an item it prefetches the next item's
//                    fp16 values into L2.
//   warps 1..8       consumers: wait on `full`, read the slot (8-byte fp16
//                    and 16-byte fp32 loads, bank-conflict free), accumulate,
//                    release the slot on `empty` (one arrival per warp).
// At the end of an item each consumer warp parks its sums in a
// double-buffered shared slot and arrives on `red_full`; consumer warp 0
// waits, adds the eight warps in order and writes the item's partial, then
// arrives on `red_empty` for that buffer.  Every wait is an mbarrier
// try_wait loop that gives up after kBulkWaitNs of global-timer time and
// raises CG_DEVFLAG_TIMEOUT; there is no CTA-wide barrier after the roles
// split, so an abandoned wait cannot deadlock the block, and the producer
// waits (bounded) for its copies still in flight before it returns.
// Requires seg_len % 8 == 0 and 16-byte aligned bases (every copy then
// starts on a 16-byte boundary and moves a multiple of 16 bytes).
constexpr int kBulkStageElems = 4096;
constexpr int kBulkConsumerWarps = 8;
constexpr int kBulkThreads = 32 * (1 + kBulkConsumerWarps);
constexpr unsigned long long kBulkWaitNs = 1000000000ull;   // 1 s

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  [[maybe_unused]] unsigned long long state;
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 %0, [%1], %2;"
               : "=l"(state)
               : "r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  [[maybe_unused]] unsigned long long state;
  asm volatile("mbarrier.arrive.shared::cta.b64 %0, [%1];" : "=l"(state) : "r"(bar) : "memory");
}

// true once the phase with the given parity has completed; false after
// limit_ns of global-timer time without completion
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity,
                                          unsigned long long limit_ns = kBulkWaitNs) {
  const unsigned long long t0 = global_ns();
  for (uint32_t it = 0;; ++it) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    if (done) return true;
    if ((it & 63u) == 63u && global_ns() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes,
                                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Bulk prefetch of [src, src + bytes) into L2 (16-byte aligned start, a
// multiple of 16 bytes); no completion to track.
__device__ __forceinline__ void bulk_prefetch_l2(const void *src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

template <int NS>
struct BulkSmem {
  float refs[NS][kBulkStageElems];
  uint16_t acts[NS][kBulkStageElems];
  unsigned long long full[NS];
  unsigned long long empty[NS];
  unsigned long long red_full[2];
  unsigned long long red_empty[2];
  float4 slot[2][kBulkConsumerWarps];
};

template <int NS>
__global__ void __launch_bounds__(kBulkThreads)
drift_bulk_kernel(const uint16_t *__restrict__ acts, const float *__restrict__ refs, uint64_t L,
                  uint64_t chunks_per_seg, uint64_t item_len, uint64_t n_items,
                  float4 *__restrict__ partials, int32_t *status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  BulkSmem<NS> &sm = *reinterpret_cast<BulkSmem<NS> *>(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < NS; ++i) {
      mbar_init((uint32_t)__cvta_generic_to_shared(&sm.full[i]), 1);
      mbar_init((uint32_t)__cvta_generic_to_shared(&sm.empty[i]), kBulkConsumerWarps);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init((uint32_t)__cvta_generic_to_shared(&sm.red_full[b]), kBulkConsumerWarps);
      mbar_init((uint32_t)__cvta_generic_to_shared(&sm.red_empty[b]), 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();   // the only CTA-wide barrier: before the roles split

  if (warp == 0) {
    // ------------------------------------------------------------- producer
    if (lane != 0) return;
    uint32_t stage = 0;
    bool ok = true;
    for (uint64_t item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const uint64_t seg = item / chunks_per_seg;
      const uint64_t ch = item - seg * chunks_per_seg;
      const uint64_t g0 = seg * L + ch * item_len;
      const uint64_t len = min(item_len, L - ch * item_len);
      // Ask L2 for the fp16 live values of this block's next item while this
      // one streams through the ring: more reads in flight than the ring holds
      // (1-2 % on every shape measured; prefetching the references as well, or
      // two items ahead, measured no better).  A hint: nothing waits on it.
      const uint64_t next = item + gridDim.x;
      if (next < n_items) {
        const uint64_t nseg = next / chunks_per_seg, nch = next - nseg * chunks_per_seg;
        const uint64_t nlen = min(item_len, L - nch * item_len);
        bulk_prefetch_l2(acts + nseg * L + nch * item_len, (uint32_t)(nlen * 2u));
      }
      for (uint64_t off = 0; off < len; off += kBulkStageElems, ++stage) {
        const uint32_t n = (uint32_t)min((uint64_t)kBulkStageElems, len - off);
        const int slot = (int)(stage % NS);
        const uint32_t round = stage / NS;
        if (round > 0 &&
            !mbar_wait((uint32_t)__cvta_generic_to_shared(&sm.empty[slot]), (round - 1) & 1u)) {
          ok = false;
          break;
        }
        const uint32_t fb = (uint32_t)__cvta_generic_to_shared(&sm.full[slot]);
        mbar_arrive_expect_tx(fb, n * 6u);
        bulk_g2s((uint32_t)__cvta_generic_to_shared(&sm.acts[slot][0]), acts + g0 + off, n * 2u, fb);
        bulk_g2s((uint32_t)__cvta_generic_to_shared(&sm.refs[slot][0]), refs + g0 + off, n * 4u, fb);
      }
    }
    if (!ok && status) atomicOr(status, CG_DEVFLAG_TIMEOUT);
    // before returning, wait (bounded) for the copies still in flight: the
    // last min(stage, NS) stages issued
    const uint32_t last = stage;
    for (uint32_t st = (last > (uint32_t)NS ? last - NS : 0); st < last; ++st) {
      const int slot = (int)(st % NS);
      if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&sm.full[slot]), (st / NS) & 1u)) {
        if (status) atomicOr(status, CG_DEVFLAG_TIMEOUT);
        break;
      }
    }
    return;
  }

  // --------------------------------------------------------------- consumers
  const int cw = warp - 1;                 // consumer warp 0..7
  const int ct = tid - 32;                 // consumer thread 0..255
  uint32_t stage = 0, local_item = 0;
  // When item_len divides L every item is item_len long and the consumers
  // skip the per-item 64-bit modulo that finds a segment's shorter last
  // item (2-2.6 % on launches of 3-stage items, where it delayed the first
  // wait of every item).
  const bool equal_items = (L % item_len) == 0;
  for (uint64_t item = blockIdx.x; item < n_items; item += gridDim.x, ++local_item) {
    const uint64_t len =
        equal_items ? item_len : min(item_len, L - (item % chunks_per_seg) * item_len);
    Acc s = {0.f, 0.f, 0.f, 0.f};
    for (uint64_t off = 0; off < len; off += kBulkStageElems, ++stage) {
      const uint32_t n = (uint32_t)min((uint64_t)kBulkStageElems, len - off);
      const int slot = (int)(stage % NS);
      // every lane waits; the warp leaves together if any lane gave up
      const bool got = mbar_wait((uint32_t)__cvta_generic_to_shared(&sm.full[slot]),
                                 (stage / NS) & 1u);
      if (!__all_sync(0xFFFFFFFFu, got)) {
        if (lane == 0 && status) atomicOr(status, CG_DEVFLAG_TIMEOUT);
        return;
      }
      const uint2 *a4 = reinterpret_cast<const uint2 *>(&sm.acts[slot][0]);
      const float4 *r4 = reinterpret_cast<const float4 *>(&sm.refs[slot][0]);
      for (uint32_t i = ct; i < n / 4; i += 32 * kBulkConsumerWarps) {
        const uint2 hv = a4[i];
        const float4 r = r4[i];
        Acc t = {0.f, 0.f, 0.f, s.m};
        const float2 h01 = half2_bits_to_float2(hv.x);
        const float2 h23 = half2_bits_to_float2(hv.y);
        acc_one(h01.x, r.x, t);
        acc_one(h01.y, r.y, t);
        acc_one(h23.x, r.z, t);
        acc_one(h23.y, r.w, t);
        s.d += t.d;
        s.e += t.e;
        s.a += t.a;
        s.m = t.m;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive((uint32_t)__cvta_generic_to_shared(&sm.empty[slot]));
    }
    // item reduction: warp tree, then warp slots summed in order by consumer warp 0
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      s.d += __shfl_down_sync(0xFFFFFFFFu, s.d, off);
      s.e += __shfl_down_sync(0xFFFFFFFFu, s.e, off);
      s.a += __shfl_down_sync(0xFFFFFFFFu, s.a, off);
      s.m = fmaxf(s.m, __shfl_down_sync(0xFFFFFFFFu, s.m, off));
    }
    const int b = (int)(local_item & 1u);
    const uint32_t use = local_item >> 1;          // how often buffer b was used before
    if (lane == 0) {
      if (use > 0 &&
          !mbar_wait((uint32_t)__cvta_generic_to_shared(&sm.red_empty[b]), (use - 1) & 1u)) {
        if (status) atomicOr(status, CG_DEVFLAG_TIMEOUT);
      }
      sm.slot[b][cw] = make_float4(s.d, s.e, s.a, s.m);
      mbar_arrive((uint32_t)__cvta_generic_to_shared(&sm.red_full[b]));
      if (cw == 0) {
        if (mbar_wait((uint32_t)__cvta_generic_to_shared(&sm.red_full[b]), use & 1u)) {
          float4 t = sm.slot[b][0];
          for (int w = 1; w < kBulkConsumerWarps; ++w) {
            const float4 v = sm.slot[b][w];
            t.x += v.x;
            t.y += v.y;
            t.z += v.z;
            t.w = fmaxf(t.w, v.w);
          }
          partials[item] = t;
        } else if (status) {
          atomicOr(status, CG_DEVFLAG_TIMEOUT);
        }
        mbar_arrive((uint32_t)__cvta_generic_to_shared(&sm.red_empty[b]));
      }
    }
    __syncwarp();
  }
}

}  // namespace

template <int NS>
static cudaError_t launch_bulk(const uint16_t *acts, const float *refs, uint64_t seg_len,
                               uint64_t cps, uint64_t item_len, uint64_t n_items,
                               float4 *partials, int32_t *status, int sm_count,
                               cudaStream_t stream) {
  const size_t smem = sizeof(BulkSmem<NS>);
  // shared-memory opt-in and occupancy, once per device
  static std::mutex mu;
  static int per_sm_of[64] = {};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  int per_sm;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (per_sm_of[dev] == 0) {
      err = cudaFuncSetAttribute(drift_bulk_kernel<NS>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (err != cudaSuccess) return err;
      int n = 0;
      err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, drift_bulk_kernel<NS>, kBulkThreads,
                                                          smem);
      if (err != cudaSuccess) return err;
      if (n < 1) return cudaErrorInvalidConfiguration;
      per_sm_of[dev] = n;
    }
    per_sm = per_sm_of[dev];
  }
  uint64_t grid = (uint64_t)sm_count * (uint64_t)per_sm;
  if (grid > n_items) grid = n_items;
  drift_bulk_kernel<NS><<<(unsigned)grid, kBulkThreads, smem, stream>>>(
      acts, refs, seg_len, cps, item_len, n_items, partials, status);
  return cudaGetLastError();
}

// Diagnostic for the bounded wait: one warp waits on a phase of an mbarrier
// that nothing arrives at.  The wait must give up after limit_ns and raise
// CG_DEVFLAG_TIMEOUT; no copy is in flight, so the block can leave.
__global__ void bounded_wait_probe_kernel(unsigned long long limit_ns, int32_t *status) {
  __shared__ __align__(8) unsigned long long bar;
  const uint32_t b = (uint32_t)__cvta_generic_to_shared(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const bool done = mbar_wait(b, 0u, limit_ns);
  if (!__all_sync(0xFFFFFFFFu, done) && threadIdx.x == 0 && status)
    atomicOr(status, CG_DEVFLAG_TIMEOUT);
}

bool drift_bulk_eligible(const uint16_t *acts, const float *refs, uint64_t seg_len) {
  return (seg_len % 8) == 0 && ((uintptr_t)acts % 16) == 0 && ((uintptr_t)refs % 16) == 0;
}

cudaError_t launch_drift_algo(const uint16_t *acts, const float *refs, uint32_t C, uint32_t S,
                              uint32_t N, uint64_t seg_len, float *scores, uint64_t stat_stride,
                              void *ws, int32_t *status, int algo, cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  const uint64_t n_seg = (uint64_t)C * S * N;
  const uint64_t cps = drift_chunks_per_seg(seg_len);
  const uint64_t item_len = drift_item_len(seg_len);
  const uint64_t n_items = n_seg * cps;
  float4 *partials = reinterpret_cast<float4 *>(static_cast<char *>(ws) + kDriftHeader);
  cudaError_t err;
  if (algo == CG_DRIFT_BULK) {
    err = launch_bulk<6>(acts, refs, seg_len, cps, item_len, n_items, partials, status,
                         info.sm_count, stream);
  } else if (algo == CG_DRIFT_BULK_2CTA) {
    err = launch_bulk<4>(acts, refs, seg_len, cps, item_len, n_items, partials, status,
                         info.sm_count, stream);
  } else {
    uint64_t grid = (uint64_t)info.sm_count * (uint64_t)info.drift_blocks_per_sm;
    if (grid > n_items) grid = n_items;
    if (grid < 1) grid = 1;
    drift_partial_kernel<<<(unsigned)grid, kDriftThreads, 0, stream>>>(acts, refs, seg_len, cps,
                                                                       item_len, n_items, partials);
    err = cudaGetLastError();
  }
  if (err != cudaSuccess) return err;
  return launch_finalize(partials, cps, C, S, N, scores, stat_stride, stream);
}

cudaError_t launch_bounded_wait_probe(uint32_t limit_us, int32_t *status, cudaStream_t stream) {
  bounded_wait_probe_kernel<<<1, 32, 0, stream>>>(1000ull * limit_us, status);
  return cudaGetLastError();
}

int drift_occupancy() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, drift_partial_kernel, kDriftThreads, 0) !=
      cudaSuccess)
    return 0;
  return n;
}

}  // namespace cg

// ----------------------------------------------------------------- no-alloc variant
// Scratch for cg_drift_scores_noalloc: the per-item partial sums live in a
// fixed device array owned by the library instead of a caller workspace.
// 262,144 float4 items = 4 MiB on each device where this module is loaded
// (its first kernel launch or first no-alloc call there), until the process
// exits.  All calls share it, so calls that overlap on the GPU (different
// streams, or other host threads) race on it.
static __device__ __align__(256) float4 g_drift_scratch[cg::kNoallocDriftItems];

namespace cg {

// Device address of g_drift_scratch on the current device.  The host-side
// symbol is only a stand-in, so the address is looked up with
// cudaGetSymbolAddress.  It is looked up on every call: the lookup is cheap
// next to a launch, and an address kept from an earlier call would point at
// freed memory after the device's context is reset and the module reloaded.
// The first lookup on a device loads the module there.
static cudaError_t noalloc_scratch(float4 **out) {
  void *p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_drift_scratch);
  if (e != cudaSuccess) return e;
  *out = static_cast<float4 *>(p);
  return cudaSuccess;
}

cudaError_t launch_drift_noalloc(const uint16_t *acts, const float *refs, uint32_t S, uint32_t N,
                                 uint64_t seg_len, float *scores, uint64_t stat_stride,
                                 cudaStream_t stream) {
  DeviceInfo info;
  if (!device_info(&info)) return cudaGetLastError();
  float4 *partials = nullptr;
  cudaError_t err = noalloc_scratch(&partials);
  if (err != cudaSuccess) return err;
  const uint64_t n_seg = (uint64_t)S * N;
  const uint64_t cps = drift_chunks_per_seg(seg_len);
  const uint64_t n_items = n_seg * cps;
  uint64_t grid = (uint64_t)info.sm_count * (uint64_t)info.drift_blocks_per_sm;
  if (grid > n_items) grid = n_items;
  if (grid < 1) grid = 1;
  drift_partial_kernel<<<(unsigned)grid, kDriftThreads, 0, stream>>>(
      acts, refs, seg_len, cps, drift_item_len(seg_len), n_items, partials);
  err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  return launch_finalize(partials, cps, 1, S, N, scores, stat_stride, stream);
}

}  // namespace cg
