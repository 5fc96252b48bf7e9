// Gaussian action noise of the appended slot, bit-exact by construction.
//
// The paper appends a slot drawn from N(0, I) after each release (Sec. 3.1).
// This library fixes the generator so every run, GPU or CPU, draws the same
// numbers:
//   Philox4x32-10 (Salmon et al., SC'11) with key (lo32(seed), hi32(seed)) and
//   counter (lo32(n), hi32(n), g, 0x4E4F4953) for action index n and the group
//   g of four action dims 4g..4g+3;
//   u = (2 (x >> 9) + 1) 2^-24, exact and inside (0, 1);
//   Box-Muller (u0,u1) -> (z0,z1), (u2,u3) -> (z2,z3): R = sqrt(-2 ln ua),
//   z = R cos(2 pi ub), z' = R sin(2 pi ub).
// ln and sincos(2 pi .) are written here as fixed sequences of individually
// rounded IEEE float32 operations (__f*_rn intrinsics: no contraction into
// fused multiply-adds, no CUDA math-library calls), so any IEEE-conforming
// implementation of the same sequence reproduces them exactly.
#pragma once

#include <stdint.h>

namespace ravel {

__device__ __forceinline__ void philox4x32_10(uint32_t& c0, uint32_t& c1, uint32_t& c2, uint32_t& c3,
                                              uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
    const uint32_t n0 = hi1 ^ c1 ^ k0;
    const uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
}

__device__ __forceinline__ float bits_to_uniform(uint32_t x) {
  // odd multiple of 2^-24 (0x33800000 is 2^-24)
  return __fmul_rn(__uint2float_rn(2u * (x >> 9) + 1u), __uint_as_float(0x33800000u));
}

// ln(u) for a positive normal float32: u = m 2^e, m in [sqrt(1/2), sqrt(2)),
// s = (m-1)/(m+1), ln m = 2 s (1 + s^2/3 + s^4/5 + s^6/7 + s^8/9),
// ln u = e ln2_hi + (e ln2_lo + ln m) with a 15-bit ln2_hi.
__device__ __forceinline__ float own_logf(float u) {
  uint32_t bits = __float_as_uint(u);
  int e = (int)((bits >> 23) & 0xFFu) - 127;
  uint32_t mb = (bits & 0x007FFFFFu) | 0x3F800000u;
  if (mb > 0x3FB504F3u) {   // m > sqrt(2): halve it
    mb -= 0x00800000u;
    e += 1;
  }
  const float m = __uint_as_float(mb);
  const float s = __fdiv_rn(__fsub_rn(m, 1.0f), __fadd_rn(m, 1.0f));
  const float s2 = __fmul_rn(s, s);
  float p = __uint_as_float(0x3DE38E39u);                          // 1/9
  p = __fadd_rn(__fmul_rn(p, s2), __uint_as_float(0x3E124925u));  // 1/7
  p = __fadd_rn(__fmul_rn(p, s2), __uint_as_float(0x3E4CCCCDu));  // 1/5
  p = __fadd_rn(__fmul_rn(p, s2), __uint_as_float(0x3EAAAAABu));  // 1/3
  p = __fadd_rn(__fmul_rn(p, s2), 1.0f);
  const float lnm = __fmul_rn(__fadd_rn(s, s), p);
  const float ef = (float)e;   // exact
  const float ln2_hi = __uint_as_float(0x3F317200u), ln2_lo = __uint_as_float(0x35BFBE8Eu);
  return __fadd_rn(__fmul_rn(ef, ln2_hi), __fadd_rn(__fmul_rn(ef, ln2_lo), lnm));
}

// (sin, cos) of 2 pi u for u in [0, 1]: x = 4u, q = rint(x), r = x - q, so that
// 2 pi u = (pi/2)(q + r) with |r| <= 1/2; Taylor polynomials of sin(pi r / 2)
// (degree 9) and cos(pi r / 2) (degree 10) in r, coefficients the correctly
// rounded float32 of (-1)^k (pi/2)^n / n!; the quadrant q mod 4 picks signs.
__device__ __forceinline__ void own_sincos2pif(float u, float* sn, float* cs) {
  const float x = __fmul_rn(u, 4.0f);
  const float q = rintf(x);
  const float r = __fsub_rn(x, q);
  const float r2 = __fmul_rn(r, r);
  float ps = __uint_as_float(0x39283C1Au);                           // n = 9
  ps = __fadd_rn(__fmul_rn(ps, r2), __uint_as_float(0xBB996966u));  // 7
  ps = __fadd_rn(__fmul_rn(ps, r2), __uint_as_float(0x3DA335E3u));  // 5
  ps = __fadd_rn(__fmul_rn(ps, r2), __uint_as_float(0xBF255DE7u));  // 3
  ps = __fadd_rn(__fmul_rn(ps, r2), __uint_as_float(0x3FC90FDBu));  // 1
  const float sr = __fmul_rn(r, ps);
  float pc = __uint_as_float(0xB7D368F9u);                           // n = 10
  pc = __fadd_rn(__fmul_rn(pc, r2), __uint_as_float(0x3A70FA83u));  // 8
  pc = __fadd_rn(__fmul_rn(pc, r2), __uint_as_float(0xBCAAE9E4u));  // 6
  pc = __fadd_rn(__fmul_rn(pc, r2), __uint_as_float(0x3E81E0F8u));  // 4
  pc = __fadd_rn(__fmul_rn(pc, r2), __uint_as_float(0xBF9DE9E6u));  // 2
  pc = __fadd_rn(__fmul_rn(pc, r2), 1.0f);                           // 0
  const float cr = pc;
  const int quad = ((int)q) & 3;
  switch (quad) {
    case 0: *sn = sr; *cs = cr; break;
    case 1: *sn = cr; *cs = -sr; break;
    case 2: *sn = -sr; *cs = -cr; break;
    default: *sn = -cr; *cs = sr; break;
  }
}

__device__ __forceinline__ void box_muller(float ua, float ub, float* z0, float* z1) {
  const float rad = __fsqrt_rn(__fmul_rn(own_logf(ua), -2.0f));
  float s, c;
  own_sincos2pif(ub, &s, &c);
  *z0 = __fmul_rn(rad, c);
  *z1 = __fmul_rn(rad, s);
}

// Four consecutive action dims 4g..4g+3 of action index n for noise seed `seed`.
__device__ __forceinline__ void action_noise4(uint64_t seed, uint64_t n, uint32_t g, float z[4]) {
  uint32_t c0 = (uint32_t)n, c1 = (uint32_t)(n >> 32), c2 = g, c3 = 0x4E4F4953u;
  philox4x32_10(c0, c1, c2, c3, (uint32_t)seed, (uint32_t)(seed >> 32));
  box_muller(bits_to_uniform(c0), bits_to_uniform(c1), &z[0], &z[1]);
  box_muller(bits_to_uniform(c2), bits_to_uniform(c3), &z[2], &z[3]);
}

}  // namespace ravel
