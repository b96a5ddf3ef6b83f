// Device generator of the ZO-Act perturbation Z (Section 3: Z ~ N(0, I)).
//
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) on
//   key = (seed_lo, seed_hi), counter = (e >> 2, layer_id, query_lo, query_hi)
// and Box-Muller on the word pairs (w0, w1), (w2, w3):
//   u1 = ((wa >> 8) + 1) * 2^-24 in (0, 1],  u2 = (wb >> 8) * 2^-24 in [0, 1)
//   za = sqrt(-2 ln u1) cos(2 pi u2),        zb = sqrt(-2 ln u1) sin(2 pi u2).
// Element e of a layer's [d_out, r] Z (e = i * r + j) is normal (e & 3) of group e >> 2.
// u1 and u2 are exact in fp32; the remaining operations are single IEEE-rounded
// library calls with no contractible multiply-add, so every kernel that includes
// this header computes bit-identical Z for the same element.
#pragma once
#include <cstdint>

namespace zoact {

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const uint32_t lo0 = 0xD2511F53u * c.x;
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

// The four raw words of group g (elements 4g .. 4g+3).
__device__ __forceinline__ uint4 z_words(uint64_t seed, uint32_t layer_id, uint64_t query, uint64_t g) {
  return philox4x32_10(make_uint4((uint32_t)g, layer_id, (uint32_t)query, (uint32_t)(query >> 32)),
                       (uint32_t)seed, (uint32_t)(seed >> 32));
}

__device__ __forceinline__ void box_muller(uint32_t wa, uint32_t wb, float& za, float& zb) {
  const float u1 = __fmul_rn((float)((wa >> 8) + 1u), 5.9604644775390625e-08f);  // exact
  const float u2 = __fmul_rn((float)(wb >> 8), 5.9604644775390625e-08f);          // exact
  const float rad = sqrtf(__fmul_rn(-2.0f, logf(u1)));
  float s, c;
  sincospif(__fmul_rn(2.0f, u2), &s, &c);                                         // sin/cos(2 pi u2)
  za = __fmul_rn(rad, c);
  zb = __fmul_rn(rad, s);
}

// Four normals of group g: elements 4g .. 4g+3 of the (seed, layer_id, query) stream.
__device__ __forceinline__ float4 z_normals4(uint64_t seed, uint32_t layer_id, uint64_t query, uint64_t g) {
  const uint4 w = z_words(seed, layer_id, query, g);
  float4 z;
  box_muller(w.x, w.y, z.x, z.y);
  box_muller(w.z, w.w, z.z, z.w);
  return z;
}

__device__ __forceinline__ float z_select(const float4& z, int i) {
  return i == 0 ? z.x : (i == 1 ? z.y : (i == 2 ? z.z : z.w));
}

}  // namespace zoact
