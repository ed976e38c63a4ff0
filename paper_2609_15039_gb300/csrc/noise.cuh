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

// ln u for u = k 2^-24, k = 1 .. 2^24: u = 2^e m with m in [sqrt(1/2), sqrt(2)) and s = m - 1
// (both exact), ln(1 + s) = s P(s) with P of degree 9 fitted to the relative error on that interval
// (least squares on Chebyshev nodes, then Lawson's reweighting toward the minimax), and
// ln u = e ln 2 + s P(s).  At most 1.6 ulp from ln u over all 2^24 inputs (checked against
// binary64), and exact (0) at u = 1.
__device__ __forceinline__ float log_unit(float u) {
  const int bits = __float_as_int(u);
  int e = (bits >> 23) - 127;
  float m = __int_as_float((bits & 0x7FFFFF) | 0x3F800000);
  if (m > 1.41421356f) {
    m = __fmul_rn(m, 0.5f);
    e += 1;
  }
  const float s = __fsub_rn(m, 1.0f);
  float p = -0.07830669730901718f;
  p = fmaf(p, s, 0.13019075989723206f);
  p = fmaf(p, s, -0.13212285935878754f);
  p = fmaf(p, s, 0.1416073590517044f);
  p = fmaf(p, s, -0.16610340774059296f);
  p = fmaf(p, s, 0.2000320553779602f);
  p = fmaf(p, s, -0.2500157058238983f);
  p = fmaf(p, s, 0.33333301544189453f);
  p = fmaf(p, s, -0.49999988079071045f);
  p = fmaf(p, s, 1.0f);
  return fmaf((float)e, 0.6931471824645996f, __fmul_rn(p, s));
}

__device__ __forceinline__ float laplace1(uint32_t r, float b) {
  const float u = __int2float_rn((int)((r & 0xFFFFFFu) + 1u)) * 0x1p-24f;  // (0, 1], exact
  const float mag = __fmul_rn(b, -log_unit(u));
  return (r >> 31) ? -mag : mag;
}

// sin(pi x) and cos(pi x) for x = 2 u2 in [0, 2), x a multiple of 2^-23: x = q / 2 + r with
// q = rint(2 x) (quarter turns) and |r| <= 1/4, both exact; sin(pi r) and cos(pi r) from their
// Taylor series to degree 9 and 10 (truncation below 3e-9 at |pi r| <= pi / 4), evaluated by
// Horner's rule in r^2; then the rotation by q quarter turns.  Error at most 1.7 ulp (checked
// against binary64 sin and cos over all 2^24 inputs), with the exact zeros of sin and cos exact.
__device__ __forceinline__ void sincospi_turns(float x, float* s, float* c) {
  const float q = rintf(2.0f * x);
  const float r = fmaf(q, -0.5f, x);
  const float r2 = __fmul_rn(r, r);
  float ps = 0.08214588661112819f;        //  pi^9 / 9!
  ps = fmaf(ps, r2, -0.5992645293207919f);  // -pi^7 / 7!
  ps = fmaf(ps, r2, 2.550164039877345f);    //  pi^5 / 5!
  ps = fmaf(ps, r2, -5.167712780049969f);   // -pi^3 / 3!
  ps = fmaf(ps, r2, 3.141592653589793f);    //  pi
  const float sr = __fmul_rn(ps, r);
  float pc = -0.02580689139001405f;         // -pi^10 / 10!
  pc = fmaf(pc, r2, 0.23533063035889312f);  //  pi^8 / 8!
  pc = fmaf(pc, r2, -1.3352627688545893f);  // -pi^6 / 6!
  pc = fmaf(pc, r2, 4.058712126416768f);    //  pi^4 / 4!
  pc = fmaf(pc, r2, -4.934802200544679f);   // -pi^2 / 2!
  pc = fmaf(pc, r2, 1.0f);
  const int t = (int)q & 3;  // (sin, cos)(pi (r + t / 2))
  *s = t == 0 ? sr : t == 1 ? pc : t == 2 ? -sr : -pc;
  *c = t == 0 ? pc : t == 1 ? -sr : t == 2 ? -pc : sr;
}

__device__ __forceinline__ void gauss2(uint32_t ra, uint32_t rb, float b, float& ea, float& eb) {
  const float u1 = __int2float_rn((int)((ra >> 8) + 1u)) * 0x1p-24f;  // (0, 1]
  const float u2 = __int2float_rn((int)(rb >> 8)) * 0x1p-24f;         // [0, 1)
  const float R = sqrtf(__fmul_rn(-2.0f, log_unit(u1)));
  float s, c;
  sincospi_turns(2.0f * u2, &s, &c);  // sin/cos of 2 pi u2; 2*u2 is exact
  const float sr = __fmul_rn(b, R);
  ea = __fmul_rn(sr, c);
  eb = __fmul_rn(sr, s);
}

template <int MECH>
__device__ __forceinline__ float4 draw_block(uint64_t j, const PhiloxKey& key, float b) {
  if (MECH == kZero) return make_float4(0.f, 0.f, 0.f, 0.f);
  const uint4 r = philox_block(j, key);
  float4 e;
  if (MECH == kLaplace) {
    e = make_float4(laplace1(r.x, b), laplace1(r.y, b), laplace1(r.z, b), laplace1(r.w, b));
  } else {
    gauss2(r.x, r.y, b, e.x, e.y);
    gauss2(r.z, r.w, b, e.z, e.w);
  }
  return e;
}

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
  return make_float4(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y), __fadd_rn(a.z, b.z), __fadd_rn(a.w, b.w));
}

}  // namespace
}  // namespace spl
