// rng.cuh -- counter-based standard-normal noise for the rollout's SAMPLE
// steps (the eps of Eq. 1), drawn where it is used: Philox4x32 with 10
// rounds (Salmon, Moraes, Dror, Shaw, SC 2011) and the Box-Muller transform.
//
// Philox4x32 maps a 128-bit counter (c0, c1, c2, c3) and a 64-bit key
// (k0, k1) to four 32-bit words; one round is
//   (hi0, lo0) = M0 c0, (hi1, lo1) = M1 c2 (64-bit products),
//   (c0, c1, c2, c3) <- (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0),
// and the key advances by (W0, W1) between rounds.
//
// Layout: element group g (elements 4g .. 4g + 3) of sample b in stream s
// (the step index) under seed K uses counter (g, b, s, 0) and key
// (K mod 2^32, K div 2^32).  A word w becomes u = (floor(w / 512) + 1/2) 2^-23
// (24 significant bits: exact in fp32, within [2^-24, 1 - 2^-24]) and the
// pairs (u0, u1), (u2, u3) become
//   sqrt(-2 ln u0) (cos 2 pi u1, sin 2 pi u1), sqrt(-2 ln u2) (cos 2 pi u3, sin 2 pi u3).
#pragma once

#include <cstdint>

namespace ff {

struct PhiloxKey {
    uint32_t k0, k1;
};

__host__ __device__ inline PhiloxKey philox_key(uint64_t seed) {
    return PhiloxKey{static_cast<uint32_t>(seed & 0xFFFFFFFFull), static_cast<uint32_t>(seed >> 32)};
}

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, PhiloxKey k) {
    constexpr uint32_t kM0 = 0xD2511F53u, kM1 = 0xCD9E8D57u;
    constexpr uint32_t kW0 = 0x9E3779B9u, kW1 = 0xBB67AE85u;
    uint32_t k0 = k.k0, k1 = k.k1;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(kM0, c.x), lo0 = kM0 * c.x;
        const uint32_t hi1 = __umulhi(kM1, c.z), lo1 = kM1 * c.z;
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
        k0 += kW0;
        k1 += kW1;
    }
    return c;
}

__device__ __forceinline__ float philox_uniform(uint32_t w) {
    return (static_cast<float>(w >> 9) + 0.5f) * 0x1p-23f;
}

// The four standard normals of element group g of sample b in stream s.
// The angle is taken as 2 pi (u - 1/2) in (-pi, pi), where the hardware sine
// and cosine are accurate to a few 1e-7 absolute (cos 2 pi u = -cos 2 pi
// (u - 1/2), likewise sin); the logarithm stays the accurate one (ln u near
// u = 1 needs relative accuracy).
__device__ __forceinline__ float4 philox_normal4(uint32_t g, uint32_t b, uint32_t s, PhiloxKey k) {
    constexpr float kTwoPi = 6.28318530717958647692f;
    const uint4 w = philox4x32_10(make_uint4(g, b, s, 0u), k);
    const float r0 = sqrtf(-2.f * logf(philox_uniform(w.x)));
    const float r1 = sqrtf(-2.f * logf(philox_uniform(w.z)));
    float s0, c0, s1, c1;
    __sincosf(kTwoPi * (philox_uniform(w.y) - 0.5f), &s0, &c0);
    __sincosf(kTwoPi * (philox_uniform(w.w) - 0.5f), &s1, &c1);
    return make_float4(-r0 * c0, -r0 * s0, -r1 * c1, -r1 * s1);
}

}  // namespace ff
