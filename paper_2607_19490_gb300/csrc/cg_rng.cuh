// cg_rng.cuh -- device-side random-number primitives of the generator.
//
// Philox4x32-10 follows the definition of Salmon, Moraes, Dror and Shaw,
// "Parallel Random Numbers: As Easy as 1, 2, 3" (SC'11): per round, two
// 32x32 -> 64-bit products of counter words 0 and 2 with the two Philox
// multipliers, the high halves XOR-ed with the other counter words and the
// round key, the key advanced by the two Weyl constants.  Normals use the
// Box-Muller transform, bounded integers Lemire's multiply-shift with
// rejection (ACM TOMACS 2019).
#pragma once

#include <stdint.h>

namespace cg {

constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

// Stream ids folded into counter word 2 as 4 * config_id + stream.
constexpr uint32_t kStreamRef = 0, kStreamNoise = 1, kStreamTamper = 2, kStreamAux = 3;
// Purposes of auxiliary word streams (counter word 1 = purpose << 24 | sub).
constexpr uint32_t kAuxOutlier = 1, kAuxStageSigma = 2, kAuxFlip = 3, kAuxControl = 4,
                   kAuxRandom = 5;

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint32_t hi0 = __umulhi(kPhiloxM0, c.x), lo0 = kPhiloxM0 * c.x;
    const uint32_t hi1 = __umulhi(kPhiloxM1, c.z), lo1 = kPhiloxM1 * c.z;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    k.x += kPhiloxW0;
    k.y += kPhiloxW1;
  }
  return c;
}

// The ten round keys of one seed, (key + r W0, key + r W1) for r = 0..9.
// They are the same for every draw of a launch, so the generator kernels take
// them precomputed (kernel parameters) and each round folds its key into the
// XOR instead of advancing it.
struct PhiloxRoundKeys {
  uint32_t k[20];
};

__device__ __forceinline__ uint4 philox4x32_10_rk(uint4 c, const PhiloxRoundKeys &rk) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint64_t p0 = (uint64_t)kPhiloxM0 * c.x;   // one 32x32 -> 64 multiply each
    const uint64_t p1 = (uint64_t)kPhiloxM1 * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ rk.k[2 * round], (uint32_t)p1,
                   (uint32_t)(p0 >> 32) ^ c.w ^ rk.k[2 * round + 1], (uint32_t)p0);
  }
  return c;
}

__device__ __forceinline__ uint2 philox_key(uint64_t seed) {
  return make_uint2((uint32_t)seed, (uint32_t)(seed >> 32));
}

// (sin, cos)(2 pi k 2^-24) for a 24-bit k.  The angle is pi t with
// t = k 2^-23, so the reduction to the nearest quarter turn q and the
// remainder r = t - q / 2 in [-1/4, 1/4] is integer arithmetic and exact.
// On the remainder, sin(pi r) and cos(pi r) are their Taylor series about 0
// through r^9 and r^10 (coefficients (-1)^j pi^(2j+1) / (2j+1)! and
// (-1)^j pi^(2j) / (2j)!); the first omitted terms are below 3e-9 and
// 1.2e-10 of the result at |r| = 1/4.  The quadrant then swaps the pair and
// sets the signs.  Over all 2^24 arguments the result is within 3.4 units
// of 2^-24 relative of the exact value.
__device__ __forceinline__ float2 sincos_2pi_u24(uint32_t k) {
  const uint32_t q = (k + (1u << 21)) >> 22;           // round(2 t), 0 .. 4
  const float r = (float)((int32_t)k - (int32_t)(q << 22)) * 0x1p-23f;
  const float r2 = r * r;
  float ps = 0.08214588661112819f;                     //  pi^9 / 9!
  ps = fmaf(ps, r2, -0.5992645293207919f);             // -pi^7 / 7!
  ps = fmaf(ps, r2, 2.550164039877345f);               //  pi^5 / 5!
  ps = fmaf(ps, r2, -5.167712780049969f);              // -pi^3 / 3!
  ps = fmaf(ps, r2, 3.141592653589793f);               //  pi
  const float sr = ps * r;                             // sin(pi r)
  float pc = -0.02580689139001405f;                    // -pi^10 / 10!
  pc = fmaf(pc, r2, 0.23533063035889312f);             //  pi^8 / 8!
  pc = fmaf(pc, r2, -1.3352627688545893f);             // -pi^6 / 6!
  pc = fmaf(pc, r2, 4.058712126416768f);               //  pi^4 / 4!
  pc = fmaf(pc, r2, -4.934802200544679f);              // -pi^2 / 2!
  const float cr = fmaf(pc, r2, 1.0f);                 // cos(pi r)
  const bool odd = q & 1u;                             // a quarter turn swaps sin and cos
  const uint32_t s_neg = (q & 2u) << 30;               // q = 2, 3: sin < 0
  const uint32_t c_neg = ((q + 1u) & 2u) << 30;        // q = 1, 2: cos < 0
  return make_float2(__uint_as_float(__float_as_uint(odd ? sr : cr) ^ c_neg),
                     __uint_as_float(__float_as_uint(odd ? cr : sr) ^ s_neg));   // (cos, sin)
}

// PTX's approximate square root (one special-function instruction).  Over
// every argument -2 ln u1 takes here it is within 2.3 units of 2^-24
// relative of the exact root, and exactly 0 at 0.
__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  asm("sqrt.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Box-Muller on two words: u1 = ((x0 >> 8) + 1) 2^-24 in (0, 1],
// u2 = (x1 >> 8) 2^-24 in [0, 1); (z0, z1) = sqrt(-2 ln u1) (cos, sin)(2 pi u2).
// u1 is exact in fp32; the angle is taken from the integer x1 >> 8.
__device__ __forceinline__ float2 box_muller(uint32_t x0, uint32_t x1) {
  const float u1 = (float)((x0 >> 8) + 1u) * 0x1p-24f;
  const float r = sqrt_approx(-2.0f * logf(u1));
  const float2 cs = sincos_2pi_u24(x1 >> 8);
  return make_float2(r * cs.x, r * cs.y);
}

// The four normals of one Philox block from precomputed round keys (counter
// word 3 = c3: 0 for every live draw, the replica index for an independent
// benign recompute).
__device__ __forceinline__ float4 normals4_rk(const PhiloxRoundKeys &rk, uint32_t q, uint32_t c1,
                                              uint32_t c2, uint32_t c3 = 0u) {
  const uint4 w = philox4x32_10_rk(make_uint4(q, c1, c2, c3), rk);
  const float2 a = box_muller(w.x, w.y);
  const float2 b = box_muller(w.z, w.w);
  return make_float4(a.x, a.y, b.x, b.y);
}

// Sequential words of an auxiliary stream (counter (i / 4, c1, c2, 0), word i % 4).
struct AuxWords {
  uint2 key;
  uint32_t c1, c2;
  uint32_t next;
  uint32_t cached;
  uint4 blk;
};

__device__ __forceinline__ AuxWords aux_words(uint64_t seed, uint32_t purpose, uint32_t sub,
                                              uint32_t config_id) {
  AuxWords w;
  w.key = philox_key(seed);
  w.c1 = (purpose << 24) | (sub & 0x00FFFFFFu);
  w.c2 = 4u * config_id + kStreamAux;
  w.next = 0;
  w.cached = 0xFFFFFFFFu;
  w.blk = make_uint4(0, 0, 0, 0);
  return w;
}

__device__ __forceinline__ uint32_t aux_next(AuxWords &w) {
  const uint32_t q = w.next >> 2;
  if (q != w.cached) {
    w.blk = philox4x32_10(make_uint4(q, w.c1, w.c2, 0u), w.key);
    w.cached = q;
  }
  const uint32_t i = w.next & 3u;
  w.next += 1;
  return i == 0 ? w.blk.x : i == 1 ? w.blk.y : i == 2 ? w.blk.z : w.blk.w;
}

// Uniform integer in [0, n), n >= 1.  Each rejection has probability below
// n / 2^32; the loop gives up after kMaxRejects draws and reports it.
constexpr int kMaxRejects = 256;
__device__ __forceinline__ uint32_t aux_bounded(AuxWords &w, uint32_t n, bool *gave_up) {
  uint64_t m = (uint64_t)aux_next(w) * (uint64_t)n;
  uint32_t low = (uint32_t)m;
  if (low < n) {
    const uint32_t threshold = (0u - n) % n;
    int tries = 0;
    while (low < threshold) {
      if (++tries > kMaxRejects) { *gave_up = true; break; }
      m = (uint64_t)aux_next(w) * (uint64_t)n;
      low = (uint32_t)m;
    }
  }
  return (uint32_t)(m >> 32);
}

}  // namespace cg
