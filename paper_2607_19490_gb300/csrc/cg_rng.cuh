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

// Box-Muller on two words: u1 = ((x0 >> 8) + 1) 2^-24 in (0, 1],
// u2 = (x1 >> 8) 2^-24 in [0, 1); (z0, z1) = sqrt(-2 ln u1) (cos, sin)(2 pi u2).
// Both uniforms are exact in fp32; sincospif takes the exact 2 u2.
__device__ __forceinline__ float2 box_muller(uint32_t x0, uint32_t x1) {
  const float u1 = (float)((x0 >> 8) + 1u) * 0x1p-24f;
  const float u2 = (float)(x1 >> 8) * 0x1p-24f;
  const float r = sqrtf(-2.0f * logf(u1));
  float s, c;
  sincospif(2.0f * u2, &s, &c);
  return make_float2(r * c, r * s);
}

// The four normals of one Philox block from precomputed round keys.
__device__ __forceinline__ float4 normals4_rk(const PhiloxRoundKeys &rk, uint32_t q, uint32_t c1,
                                              uint32_t c2, uint32_t c3 = 0u) {
  const uint4 w = philox4x32_10_rk(make_uint4(q, c1, c2, c3), rk);
  const float2 a = box_muller(w.x, w.y);
  const float2 b = box_muller(w.z, w.w);
  return make_float4(a.x, a.y, b.x, b.y);
}

// The four normals of one Philox block (counter word 3 = c3: 0 for every
// live draw, the replica index for an independent benign recompute).
__device__ __forceinline__ float4 normals4(uint2 key, uint32_t q, uint32_t c1, uint32_t c2,
                                           uint32_t c3 = 0u) {
  const uint4 w = philox4x32_10(make_uint4(q, c1, c2, c3), key);
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
