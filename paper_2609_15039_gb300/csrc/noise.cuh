// Noise draw shared by the mask kernels (elementwise.cu) and the decode product's fused mask
// (gemv.cu): Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11, Sec. 3.3) and the Laplace /
// Gaussian transforms at scale Delta f / eps (Sec. 4.4).  Element e of a flat [rows, cols]
// tensor is lane e % 4 of Philox block e / 4 + offset, key = seed, counter words 2-3 =
// stream_id.  The mask is one fp32 round-to-nearest addition x + eta (Sec. 3.3.1).
#pragma once

#include <cstdint>

#include <cuda_runtime.h>

namespace spl {
namespace {

constexpr uint32_t kPhiloxM0 = 0xD2511F53u;  // round multiplier for counter word 0
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;  // round multiplier for counter word 2
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;  // key increment, word 0
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;  // key increment, word 1

// The round keys and counter words 2-3 of one (seed, stream_id), computed once on the host:
// round r uses the key (lo(seed) + r W0, hi(seed) + r W1) mod 2^32.  A kernel receives them as a
// __grid_constant__ parameter, so every round's key enters its XOR straight from the constant
// bank, with no addition per round.
struct PhiloxKey {
  uint32_t k0[10], k1[10];
  uint32_t s0, s1;
};

inline PhiloxKey make_philox_key(uint64_t seed, uint64_t stream_id) {
  PhiloxKey k;
  uint32_t a = (uint32_t)seed, b = (uint32_t)(seed >> 32);
  for (int r = 0; r < 10; ++r) {
    k.k0[r] = a;
    k.k1[r] = b;
    a += kPhiloxW0;
    b += kPhiloxW1;
  }
  k.s0 = (uint32_t)stream_id;
  k.s1 = (uint32_t)(stream_id >> 32);
  return k;
}

// Philox4x32-10 of counter (lo j, hi j, s0, s1).
__device__ __forceinline__ uint4 philox_block(uint64_t j, const PhiloxKey& key) {
  uint4 c = make_uint4((uint32_t)j, (uint32_t)(j >> 32), key.s0, key.s1);
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t hi0 = __umulhi(kPhiloxM0, c.x), lo0 = kPhiloxM0 * c.x;
    const uint32_t hi1 = __umulhi(kPhiloxM1, c.z), lo1 = kPhiloxM1 * c.z;
    c = make_uint4(hi1 ^ c.y ^ key.k0[r], lo1, hi0 ^ c.w ^ key.k1[r], lo0);
  }
  return c;
}

enum { kLaplace = 0, kGaussian = 1, kZero = 2 };

// Packed pairs of fp32: one fma.rn.f32x2 does the two round-to-nearest FMAs that two fmaf calls
// would, so a pair of uniforms (or angles) runs its polynomial in one chain, same results.
__device__ __forceinline__ unsigned long long p2(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void up2(unsigned long long v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ unsigned long long fma2(unsigned long long a, unsigned long long b, unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ unsigned long long fma2c(unsigned long long a, unsigned long long b, float c) {
  return fma2(a, b, p2(c, c));
}

// ln u for u = k 2^-24, k = 1 .. 2^24: u = 2^e m with m in (sqrt(1/2), sqrt(2)] and s = m - 1
// (both exact), ln(1 + s) = s P(s) with P of degree 9 fitted to the relative error on that interval
// (least squares on Chebyshev nodes, then Lawson's reweighting toward the minimax), and
// ln u = e ln 2 + s P(s).  At most 1.6 ulp from ln u over all 2^24 inputs (checked against
// binary64), and exact (0) at u = 1.  The reduction is the usual branch-free one on the bit
// pattern: subtracting the bits of the float just above sqrt(1/2) leaves e in the high bits
// (arithmetic shift) and, added back to the low 23 bits, the bits of m.
// Two uniforms at once: ln u0 and ln u1.
__device__ __forceinline__ void log_unit2(float u0, float u1, float& l0, float& l1) {
  constexpr int kOff = 0x3F3504F4;  // bits of the float just above sqrt(1/2)
  const int d0 = __float_as_int(u0) - kOff, d1 = __float_as_int(u1) - kOff;
  const float m0 = __int_as_float((d0 & 0x7FFFFF) + kOff), m1 = __int_as_float((d1 & 0x7FFFFF) + kOff);
  const unsigned long long s = p2(__fsub_rn(m0, 1.0f), __fsub_rn(m1, 1.0f));
  unsigned long long p = p2(-0.07830669730901718f, -0.07830669730901718f);
  p = fma2c(p, s, 0.13019075989723206f);
  p = fma2c(p, s, -0.13212285935878754f);
  p = fma2c(p, s, 0.1416073590517044f);
  p = fma2c(p, s, -0.16610340774059296f);
  p = fma2c(p, s, 0.2000320553779602f);
  p = fma2c(p, s, -0.2500157058238983f);
  p = fma2c(p, s, 0.33333301544189453f);
  p = fma2c(p, s, -0.49999988079071045f);
  p = fma2c(p, s, 1.0f);
  const unsigned long long ps = fma2c(p, s, -0.0f);  // fl(p s): adding -0 changes no rounding
  up2(fma2(p2((float)(d0 >> 23), (float)(d1 >> 23)), p2(0.6931471824645996f, 0.6931471824645996f), ps), l0, l1);
}

// sin(pi x) and cos(pi x) for x = 2 u2 in [0, 2), x a multiple of 2^-23: x = q / 2 + r with
// q = rint(2 x) (quarter turns) and |r| <= 1/4, both exact; sin(pi r) and cos(pi r) from their
// Taylor series to degree 9 and 10 (truncation below 3e-9 at |pi r| <= pi / 4), evaluated by
// Horner's rule in r^2; then the rotation by q quarter turns.  Error at most 1.7 ulp (checked
// against binary64 sin and cos over all 2^24 inputs), with the exact zeros of sin and cos exact.
// Two angles at once.
__device__ __forceinline__ void sincospi_turns2(float x0, float x1, float* s0, float* c0, float* s1, float* c1) {
  const float q0 = rintf(2.0f * x0), q1 = rintf(2.0f * x1);
  const float r0 = fmaf(q0, -0.5f, x0), r1 = fmaf(q1, -0.5f, x1);
  const unsigned long long r = p2(r0, r1), r2 = p2(__fmul_rn(r0, r0), __fmul_rn(r1, r1));
  unsigned long long ps = p2(0.08214588661112819f, 0.08214588661112819f);
  ps = fma2c(ps, r2, -0.5992645293207919f);
  ps = fma2c(ps, r2, 2.550164039877345f);
  ps = fma2c(ps, r2, -5.167712780049969f);
  ps = fma2c(ps, r2, 3.141592653589793f);
  float sr0, sr1;
  up2(fma2c(ps, r, -0.0f), sr0, sr1);  // fl(ps r)
  unsigned long long pc = p2(-0.02580689139001405f, -0.02580689139001405f);
  pc = fma2c(pc, r2, 0.23533063035889312f);
  pc = fma2c(pc, r2, -1.3352627688545893f);
  pc = fma2c(pc, r2, 4.058712126416768f);
  pc = fma2c(pc, r2, -4.934802200544679f);
  pc = fma2c(pc, r2, 1.0f);
  float pc0, pc1;
  up2(pc, pc0, pc1);
  // quarter turn t: (sin, cos) = (sr, pc), (pc, -sr), (-sr, -pc), (-pc, sr) for t mod 4 = 0..3;
  // odd t swaps the two, t = 2, 3 negates the sine and t = 1, 2 the cosine (sign-bit flips)
  const uint32_t t0 = (uint32_t)(int)q0, t1 = (uint32_t)(int)q1;
  *s0 = __uint_as_float(__float_as_uint((t0 & 1u) ? pc0 : sr0) ^ ((t0 & 2u) << 30));
  *c0 = __uint_as_float(__float_as_uint((t0 & 1u) ? sr0 : pc0) ^ (((t0 + 1u) & 2u) << 30));
  *s1 = __uint_as_float(__float_as_uint((t1 & 1u) ? pc1 : sr1) ^ ((t1 & 2u) << 30));
  *c1 = __uint_as_float(__float_as_uint((t1 & 1u) ? sr1 : pc1) ^ (((t1 + 1u) & 2u) << 30));
}

// The hardware square-root approximation (sqrt.approx.f32), no Newton refinement: at most
// 1.68 x 2^-24 relative error over every float in [1, 4) and over all 2^24 values of -2 ln u
// the draw can take (measured against binary64 on GB300), against 2^-24 for the rounded root.
__device__ __forceinline__ float sqrt_approx(float x) {
  float r;
  asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

template <int MECH>
__device__ __forceinline__ float4 draw_block(uint64_t j, const PhiloxKey& key, float b) {
  if (MECH == kZero) return make_float4(0.f, 0.f, 0.f, 0.f);
  const uint4 r = philox_block(j, key);
  float4 e;
  if (MECH == kLaplace) {
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
    float u[4], l[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) u[i] = __int2float_rn((int)((w[i] & 0xFFFFFFu) + 1u)) * 0x1p-24f;
    log_unit2(u[0], u[1], l[0], l[1]);
    log_unit2(u[2], u[3], l[2], l[3]);
    float m[4];  // b (-ln u), two at a time; the sign is the top bit of the word
    up2(fma2(p2(-b, -b), p2(l[0], l[1]), p2(-0.0f, -0.0f)), m[0], m[1]);
    up2(fma2(p2(-b, -b), p2(l[2], l[3]), p2(-0.0f, -0.0f)), m[2], m[3]);
    float v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = __uint_as_float(__float_as_uint(m[i]) ^ (w[i] & 0x80000000u));
    e = make_float4(v[0], v[1], v[2], v[3]);
  } else {  // Box-Muller on the pairs (x, y) and (z, w), the two done side by side
    const float ua = __int2float_rn((int)((r.x >> 8) + 1u)) * 0x1p-24f;  // (0, 1]
    const float ub = __int2float_rn((int)((r.z >> 8) + 1u)) * 0x1p-24f;
    const float va = __int2float_rn((int)(r.y >> 8)) * 0x1p-24f;         // [0, 1)
    const float vb = __int2float_rn((int)(r.w >> 8)) * 0x1p-24f;
    float la, lb, sa, ca, sb, cb;
    log_unit2(ua, ub, la, lb);
    sincospi_turns2(2.0f * va, 2.0f * vb, &sa, &ca, &sb, &cb);  // sin/cos of 2 pi v; 2 v is exact
    float ra_, rb_;  // b sqrt(-2 ln u) for both pairs (-2 ln u is exact)
    up2(fma2(p2(b, b), p2(sqrt_approx(-2.0f * la), sqrt_approx(-2.0f * lb)), p2(-0.0f, -0.0f)), ra_, rb_);
    float x0, y0, x1, y1;
    up2(fma2(p2(ra_, ra_), p2(ca, sa), p2(-0.0f, -0.0f)), x0, y0);
    up2(fma2(p2(rb_, rb_), p2(cb, sb), p2(-0.0f, -0.0f)), x1, y1);
    e = make_float4(x0, y0, x1, y1);
  }
  return e;
}

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
  return make_float4(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y), __fadd_rn(a.z, b.z), __fadd_rn(a.w, b.w));
}

}  // namespace
}  // namespace spl
