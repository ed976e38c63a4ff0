// a2 noise, a3 mask, a6 unmask and the TF32 split: bandwidth-bound elementwise
// kernels over flat fp32 tensors.
//
// Noise follows the Gaussian mechanism N(0, (Delta f/eps)^2 I) of Sec. 4.4
// (Prop. eps-GDP mechanism) or the Laplace variant at the same scale, drawn
// from Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11, Sec. 3.3).  The mask
// is x~ = x + eta (Sec. 3.3.1) and the unmask r - W eta (Eq.
// add-and-then-subtract), each one fp32 round-to-nearest operation: the
// explicit __fadd_rn/__fsub_rn/__fmul_rn keep the compiler from contracting
// them into an FMA, so the eta written to N is exactly the eta added to x.
//
// Layout: one thread handles one Philox block (4 consecutive elements) per
// step as a float4; two blocks are in flight per loop trip.  The grid is a
// whole number of waves over the SMs (grid-stride loop).

#include <algorithm>

#include <cuda_fp16.h>

#include "common.cuh"
#include "noise.cuh"

namespace spl {
namespace {

constexpr int kThreads = 256;

// xt = x + eta (if xt), nout = eta (if nout).  n elements, nb = ceil(n/4) Philox blocks.
template <int MECH>
__global__ void __launch_bounds__(kThreads) noise_mask_kernel(float* xt, float* __restrict__ nout,
                                                              const float* x, int64_t n, float b,
                                                              const __grid_constant__ PhiloxKey key,
                                                              uint64_t offset_host, const uint64_t* offset_dev) {
  pdl_wait();
  pdl_trigger();
  const uint64_t offset = offset_host + (offset_dev ? *offset_dev : 0ull);
  const int64_t nb_full = n >> 2;  // blocks with all 4 elements in range
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const float4* x4 = reinterpret_cast<const float4*>(x);
  float4* xt4 = reinterpret_cast<float4*>(xt);
  float4* n4 = reinterpret_cast<float4*>(nout);
  // two blocks per trip: issue both loads first
  for (; i + stride < nb_full; i += 2 * stride) {
    float4 xa, xb;
    if (xt) {
      xa = __ldcs(x4 + i);
      xb = __ldcs(x4 + i + stride);
    }
    const float4 ea = draw_block<MECH>((uint64_t)i + offset, key, b);
    const float4 eb = draw_block<MECH>((uint64_t)(i + stride) + offset, key, b);
    if (nout) {
      __stcs(n4 + i, ea);
      __stcs(n4 + i + stride, eb);
    }
    if (xt) {
      __stcs(xt4 + i, add4(xa, ea));
      __stcs(xt4 + i + stride, add4(xb, eb));
    }
  }
  for (; i < nb_full; i += stride) {
    const float4 e = draw_block<MECH>((uint64_t)i + offset, key, b);
    if (nout) __stcs(n4 + i, e);
    if (xt) __stcs(xt4 + i, add4(__ldcs(x4 + i), e));
  }
  // ragged tail: the last, partial Philox block
  if (blockIdx.x == 0 && threadIdx.x == 0 && (n & 3)) {
    const int64_t j = nb_full;
    const float4 e = draw_block<MECH>((uint64_t)j + offset, key, b);
    const float ev[4] = {e.x, e.y, e.z, e.w};
    for (int l = 0; l < (int)(n & 3); ++l) {
      const int64_t idx = 4 * j + l;
      if (nout) nout[idx] = ev[l];
      if (xt) xt[idx] = __fadd_rn(x[idx], ev[l]);
    }
  }
}

__global__ void rng_advance_kernel(uint64_t* offset_dev, uint64_t delta) {
  pdl_wait();
  pdl_trigger();
  *offset_dev += delta;
}

// Binary64 mask (Sec. 5.5): xt = fl64((double)x + (double)eta) with eta drawn exactly as above:
// one rounding of at most 2^-53 |xt| (none at all while the exponents of x and eta are within 29).
template <int MECH>
__global__ void __launch_bounds__(kThreads) noise_mask_f64_kernel(double* __restrict__ xt, const float* __restrict__ x,
                                                                  int64_t n, float b, const __grid_constant__ PhiloxKey key, uint64_t offset_host,
                                                                  const uint64_t* offset_dev) {
  pdl_wait();
  pdl_trigger();
  const uint64_t offset = offset_host + (offset_dev ? *offset_dev : 0ull);
  const int64_t nb = (n + 3) >> 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nb; i += stride) {
    const float4 e = draw_block<MECH>((uint64_t)i + offset, key, b);
    const float ev[4] = {e.x, e.y, e.z, e.w};
    if (4 * i + 3 < n) {
      const float4 xv = __ldcs(reinterpret_cast<const float4*>(x) + i);
      double2* o = reinterpret_cast<double2*>(xt + 4 * i);
      __stcs(o, make_double2((double)xv.x + (double)ev[0], (double)xv.y + (double)ev[1]));
      __stcs(o + 1, make_double2((double)xv.z + (double)ev[2], (double)xv.w + (double)ev[3]));
    } else {
      for (int l = 0; l < 4 && 4 * i + l < n; ++l) xt[4 * i + l] = (double)x[4 * i + l] + (double)ev[l];
    }
  }
}

// Slalom comparator (Sec. 6.2): fixed point with 8 fractional bits, mask uniform in Z_q,
// q = 2^23 + 2^21 + 7.  Element e draws block e / 2 + offset and takes words 2 (e % 2) and
// 2 (e % 2) + 1 as the 64-bit integer lo + 2^32 hi; eta = that mod q.  Values below 2^24 are
// exact in fp32, so the field elements travel as fp32.
constexpr int64_t kSlalomQ = (1 << 23) + (1 << 21) + 7;

__device__ __forceinline__ float slalom_mask1(float x, uint32_t lo, uint32_t hi, float* eta_out) {
  const int64_t eta = (int64_t)((((uint64_t)hi << 32) | lo) % (uint64_t)kSlalomQ);
  const int64_t xq = ((int64_t)llrintf(x * 256.0f) % kSlalomQ + kSlalomQ) % kSlalomQ;
  if (eta_out) *eta_out = (float)eta;
  return (float)((xq + eta) % kSlalomQ);
}

__global__ void __launch_bounds__(kThreads) slalom_mask_kernel(float* __restrict__ xt, float* __restrict__ eta,
                                                               const float* __restrict__ x, int64_t n, const __grid_constant__ PhiloxKey key,
                                                               uint64_t offset) {
  pdl_wait();
  pdl_trigger();
  const int64_t nb = (n + 1) >> 1;  // two elements per Philox block
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nb; i += stride) {
    const uint64_t j = (uint64_t)i + offset;
    const uint4 r = philox_block(j, key);
    const int64_t e = 2 * i;
    xt[e] = slalom_mask1(x[e], r.x, r.y, eta ? eta + e : nullptr);
    if (e + 1 < n) xt[e + 1] = slalom_mask1(x[e + 1], r.z, r.w, eta ? eta + e + 1 : nullptr);
  }
}

__global__ void __launch_bounds__(kThreads) slalom_quantize_kernel(float* __restrict__ out,
                                                                   const float* __restrict__ v, int64_t n) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    out[i] = rintf(v[i] * 256.0f);  // v 2^8 is exact; rint rounds half to even
}

// The raw Philox words of the stream (element e = lane e % 4 of block e / 4 + offset).
__global__ void __launch_bounds__(kThreads) random_bits_kernel(uint32_t* __restrict__ out, int64_t n, const __grid_constant__ PhiloxKey key,
                                                               uint64_t offset_host, const uint64_t* offset_dev) {
  pdl_wait();
  pdl_trigger();
  const uint64_t offset = offset_host + (offset_dev ? *offset_dev : 0ull);
  const int64_t nb = (n + 3) >> 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nb; i += stride) {
    const uint64_t j = (uint64_t)i + offset;
    const uint4 r = philox_block(j, key);
    if (4 * i + 3 < n) {
      reinterpret_cast<uint4*>(out)[i] = r;
    } else {
      const uint32_t rv[4] = {r.x, r.y, r.z, r.w};
      for (int l = 0; l < 4 && 4 * i + l < n; ++l) out[4 * i + l] = rv[l];
    }
  }
}

// out = a + s * b elementwise with s = +1 (mask) or -1 (unmask), one rounding.
template <bool SUB>
__global__ void __launch_bounds__(kThreads) addsub_kernel(float* out, const float* a,
                                                          const float* __restrict__ b, int64_t n) {
  const int64_t n4 = n >> 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const float4* a4 = reinterpret_cast<const float4*>(a);
  const float4* b4 = reinterpret_cast<const float4*>(b);
  float4* o4 = reinterpret_cast<float4*>(out);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 x = __ldcs(a4 + i), y = __ldcs(b4 + i);
    float4 r;
    if (SUB) {
      r = make_float4(__fsub_rn(x.x, y.x), __fsub_rn(x.y, y.y), __fsub_rn(x.z, y.z), __fsub_rn(x.w, y.w));
    } else {
      r = add4(x, y);
    }
    __stcs(o4 + i, r);
  }
  if (blockIdx.x == 0 && threadIdx.x < (n & 3)) {
    const int64_t idx = 4 * n4 + threadIdx.x;
    out[idx] = SUB ? __fsub_rn(a[idx], b[idx]) : __fadd_rn(a[idx], b[idx]);
  }
}

__device__ __forceinline__ float tf32_rna(float v) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(v));
  return __uint_as_float(r);
}

__global__ void __launch_bounds__(kThreads) split_tf32_kernel(float* __restrict__ hi, float* __restrict__ lo,
                                                              const float* __restrict__ src, int64_t n) {
  pdl_wait();
  pdl_trigger();
  const int64_t n4 = n >> 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const float4* s4 = reinterpret_cast<const float4*>(src);
  float4* h4 = reinterpret_cast<float4*>(hi);
  float4* l4 = reinterpret_cast<float4*>(lo);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 v = __ldcs(s4 + i);
    const float4 h = make_float4(tf32_rna(v.x), tf32_rna(v.y), tf32_rna(v.z), tf32_rna(v.w));
    h4[i] = h;
    l4[i] = make_float4(__fsub_rn(v.x, h.x), __fsub_rn(v.y, h.y), __fsub_rn(v.z, h.z), __fsub_rn(v.w, h.w));
  }
  if (blockIdx.x == 0 && threadIdx.x < (n & 3)) {
    const int64_t idx = 4 * n4 + threadIdx.x;
    const float h = tf32_rna(src[idx]);
    hi[idx] = h;
    lo[idx] = __fsub_rn(src[idx], h);
  }
}

// fp16 split of a row-major matrix, one block per row: e = fp16_row_exponent(max |x|) brings the
// row's largest entry into [2^14, 2^15); hi = fp16(x 2^e), lo = fp16(x 2^e - hi) (the difference
// is exact in fp32).  cols % 8 == 0; each thread handles 8 consecutive entries at a time, and the
// second pass re-reads the row from L1.
__global__ void __launch_bounds__(kThreads) split_fp16_kernel(uint16_t* __restrict__ hi, uint16_t* __restrict__ lo,
                                                              int* __restrict__ row_exp, const float* __restrict__ src,
                                                              int64_t cols) {
  pdl_trigger();  // before waiting: see the split kernel below
  pdl_wait();  // src may come from the kernel before this one, which may still read hi and lo
  __shared__ float warp_max[kThreads / 32];
  const int64_t r = blockIdx.x;
  const float4* row = reinterpret_cast<const float4*>(src + r * cols);
  const int64_t q = cols >> 2;
  float m0 = 0.f, m1 = 0.f;
  int64_t i = threadIdx.x;
  for (; i + kThreads < q; i += 2 * kThreads) {
    const float4 a = row[i], b = row[i + kThreads];
    m0 = fmaxf(m0, fmaxf(fmaxf(fabsf(a.x), fabsf(a.y)), fmaxf(fabsf(a.z), fabsf(a.w))));
    m1 = fmaxf(m1, fmaxf(fmaxf(fabsf(b.x), fabsf(b.y)), fmaxf(fabsf(b.z), fabsf(b.w))));
  }
  if (i < q) {
    const float4 a = row[i];
    m0 = fmaxf(m0, fmaxf(fmaxf(fabsf(a.x), fabsf(a.y)), fmaxf(fabsf(a.z), fabsf(a.w))));
  }
  float m = fmaxf(m0, m1);
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  m = warp_max[0];
#pragma unroll
  for (int w = 1; w < kThreads / 32; ++w) m = fmaxf(m, warp_max[w]);
  const int e = fp16_row_exponent(m);
  if (threadIdx.x == 0) row_exp[r] = e;
  const float sc = __int_as_float((e + 127) << 23);
  uint4* h8 = reinterpret_cast<uint4*>(hi + r * cols);
  uint4* l8 = reinterpret_cast<uint4*>(lo + r * cols);
  for (int64_t c = threadIdx.x; c < (cols >> 3); c += kThreads) {
    const float4 a = row[2 * c], b = row[2 * c + 1];
    const float xs[8] = {a.x * sc, a.y * sc, a.z * sc, a.w * sc, b.x * sc, b.y * sc, b.z * sc, b.w * sc};
    __align__(16) __half h[8];
    __align__(16) __half l[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      h[k] = __float2half_rn(xs[k]);
      l[k] = __float2half_rn(__fsub_rn(xs[k], __half2float(h[k])));
    }
    h8[c] = *reinterpret_cast<const uint4*>(h);
    l8[c] = *reinterpret_cast<const uint4*>(l);
  }
}

// The same split with the row held in registers: one block per row, CH chunks of 8 entries per
// thread, all loads issued before any is used, so a row costs one memory round trip.
// MECH >= 0: the row is first masked (a2 + a3 fused into the split): xt = fl32(x + eta) with eta
// drawn exactly as noise_mask_kernel draws it (element e: lane e % 4 of Philox block e / 4 +
// offset), written to xt_out when it is not NULL, then split.  MECH == kStored: eta is read
// from `stored` (a noise drawn earlier, e.g. with a bank of corrections), xt = fl32(x + eta).
constexpr int kNoMask = -1;
constexpr int kStored = 3;

template <int CH, int MECH>
__global__ void __launch_bounds__(kThreads) split_fp16_regs_kernel(uint16_t* __restrict__ hi,
                                                                   uint16_t* __restrict__ lo,
                                                                   int* __restrict__ row_exp,
                                                                   const float* __restrict__ src, int64_t cols,
                                                                   float* __restrict__ xt_out, float b, const __grid_constant__ PhiloxKey key,
                                                                   uint64_t offset_host, const uint64_t* offset_dev,
                                                                   const float* __restrict__ stored, int64_t x_rows,
                                                                   uint64_t noise_delta) {
  // The product after this split may be scheduled before the split waits: every block of this
  // grid has started by then, and so has every CTA of the kernel it waits for, so the product's
  // CTAs (which read only the weight before they wait, an L2 prefetch of C aside) take SMs that
  // nothing before them still needs; they stream the weight while the kernel before this split ends.
  pdl_trigger();
  pdl_wait();
  __shared__ float warp_max[kThreads / 32];
  const int64_t r = blockIdx.x;
  // rows from x_rows on (and every row when src is NULL, with a mechanism) are the noise alone,
  // drawn noise_delta Philox blocks further on, their counters starting again at row x_rows
  const bool own = r < x_rows;
  const float4* row = (src && own) ? reinterpret_cast<const float4*>(src + r * cols) : nullptr;
  const int64_t n8 = cols >> 3;
  float4 v[2 * CH];
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    const int64_t i = threadIdx.x + (int64_t)c * kThreads;
    if (row && i < n8) {
      v[2 * c] = __ldg(row + 2 * i);
      v[2 * c + 1] = __ldg(row + 2 * i + 1);
    } else {
      v[2 * c] = v[2 * c + 1] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  if constexpr (MECH == kStored) {
    const float4* nrow = reinterpret_cast<const float4*>(stored + r * cols);
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const int64_t i = threadIdx.x + (int64_t)c * kThreads;
      if (i >= n8) break;
      v[2 * c] = add4(v[2 * c], __ldg(nrow + 2 * i));
      v[2 * c + 1] = add4(v[2 * c + 1], __ldg(nrow + 2 * i + 1));
      if (xt_out) {
        float4* o = reinterpret_cast<float4*>(xt_out + r * cols);
        __stcs(o + 2 * i, v[2 * c]);
        __stcs(o + 2 * i + 1, v[2 * c + 1]);
      }
    }
  } else if constexpr (MECH != kNoMask) {
    const uint64_t offset = offset_host + (offset_dev ? *offset_dev : 0ull) + (own ? 0ull : noise_delta);
    const int64_t rr = own ? r : r - x_rows;
    const uint64_t j0 = (uint64_t)((rr * cols) >> 2) + offset;  // cols % 8 == 0: rows start on a block
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const int64_t i = threadIdx.x + (int64_t)c * kThreads;
      if (i >= n8) break;
      const uint64_t j = j0 + 2 * (uint64_t)i;
      const float4 e0 = draw_block<MECH>(j, key, b), e1 = draw_block<MECH>(j + 1, key, b);
      v[2 * c] = row ? add4(v[2 * c], e0) : e0;
      v[2 * c + 1] = row ? add4(v[2 * c + 1], e1) : e1;
      if (xt_out) {
        float4* o = reinterpret_cast<float4*>(xt_out + r * cols);
        __stcs(o + 2 * i, v[2 * c]);
        __stcs(o + 2 * i + 1, v[2 * c + 1]);
      }
    }
  }
  float m = 0.f;
#pragma unroll
  for (int c = 0; c < 2 * CH; ++c)
    m = fmaxf(m, fmaxf(fmaxf(fabsf(v[c].x), fabsf(v[c].y)), fmaxf(fabsf(v[c].z), fabsf(v[c].w))));
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  m = warp_max[0];
#pragma unroll
  for (int w = 1; w < kThreads / 32; ++w) m = fmaxf(m, warp_max[w]);
  const int e = fp16_row_exponent(m);
  if (threadIdx.x == 0) row_exp[r] = e;
  const float sc = __int_as_float((e + 127) << 23);
  uint4* h8 = reinterpret_cast<uint4*>(hi + r * cols);
  uint4* l8 = reinterpret_cast<uint4*>(lo + r * cols);
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    const int64_t i = threadIdx.x + (int64_t)c * kThreads;
    if (i >= n8) break;
    const float4 a = v[2 * c], bb = v[2 * c + 1];
    const float xs[8] = {a.x * sc, a.y * sc, a.z * sc, a.w * sc, bb.x * sc, bb.y * sc, bb.z * sc, bb.w * sc};
    __align__(16) __half h[8];
    __align__(16) __half l[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      h[k] = __float2half_rn(xs[k]);
      l[k] = __float2half_rn(__fsub_rn(xs[k], __half2float(h[k])));
    }
    h8[i] = *reinterpret_cast<const uint4*>(h);
    l8[i] = *reinterpret_cast<const uint4*>(l);
  }
}

int grid_for(int64_t work_items, int blocks_per_sm) {
  const int64_t want = ceil_div(work_items, kThreads);
  const int64_t cap = (int64_t)device_sm_count() * blocks_per_sm;
  return (int)std::max<int64_t>(1, std::min(want, cap));
}

spl_status launch_noise_mask(float* xt, float* nout, const float* x, int64_t n, double sensitivity, double eps,
                             spl_mech mech, spl_rng rng, cudaStream_t stream) {
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  const float b = std::isinf(eps) ? 0.0f : (float)(sensitivity / eps);
  const int grid = grid_for(ceil_div(n, 4), 8);
  const PhiloxKey key = make_philox_key(rng.seed, rng.stream_id);
  if (b == 0.0f) {
    return launch_pdl(noise_mask_kernel<kZero>, dim3(grid), dim3(kThreads), 0, stream, xt, nout, x, n, b, key, rng.offset, rng.offset_dev);
  } else if (mech == SPL_MECH_LAPLACE) {
    return launch_pdl(noise_mask_kernel<kLaplace>, dim3(grid), dim3(kThreads), 0, stream, xt, nout, x, n, b, key, rng.offset, rng.offset_dev);
  } else {
    return launch_pdl(noise_mask_kernel<kGaussian>, dim3(grid), dim3(kThreads), 0, stream, xt, nout, x, n, b, key, rng.offset, rng.offset_dev);
  }
}

}  // namespace

spl_status validate_noise(int64_t rows, int64_t cols, double sensitivity, double eps, spl_mech mech) {
  if (rows < 0 || cols < 0) return SPL_EINVAL;
  if (!(eps > 0.0)) return SPL_EINVAL;  // also rejects NaN
  if (!(sensitivity >= 0.0) || std::isinf(sensitivity)) return SPL_EINVAL;
  if (mech != SPL_MECH_LAPLACE && mech != SPL_MECH_GAUSSIAN) return SPL_EINVAL;
  return SPL_OK;
}

// Row split with an optional fused mask (mech < 0: none).  Rows whose register copy does not fit
// (more than 16384 entries) and no mask take the two-pass kernel.
template <int MECH>
spl_status launch_split_rows(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* src, int64_t rows,
                             int64_t cols, float* xt_out, float b, const spl_rng& rng, cudaStream_t stream,
                             const float* stored = nullptr, int64_t x_rows = -1, uint64_t noise_delta = 0) {
  if (x_rows < 0) x_rows = rows;
  const int64_t per_thread = ceil_div(cols >> 3, kThreads);  // chunks of 8 per thread
  const dim3 grid((unsigned)rows), block(kThreads);
  const PhiloxKey key = make_philox_key(rng.seed, rng.stream_id);
  if (per_thread <= 1)
    return launch_pdl(split_fp16_regs_kernel<1, MECH>, grid, block, 0, stream, hi, lo, row_exp, src, cols, xt_out, b,
                      key, rng.offset, rng.offset_dev, stored, x_rows, noise_delta);
  if (per_thread <= 2)
    return launch_pdl(split_fp16_regs_kernel<2, MECH>, grid, block, 0, stream, hi, lo, row_exp, src, cols, xt_out, b,
                      key, rng.offset, rng.offset_dev, stored, x_rows, noise_delta);
  if (per_thread <= 4)
    return launch_pdl(split_fp16_regs_kernel<4, MECH>, grid, block, 0, stream, hi, lo, row_exp, src, cols, xt_out, b,
                      key, rng.offset, rng.offset_dev, stored, x_rows, noise_delta);
  if (per_thread <= 8)
    return launch_pdl(split_fp16_regs_kernel<8, MECH>, grid, block, 0, stream, hi, lo, row_exp, src, cols, xt_out, b,
                      key, rng.offset, rng.offset_dev, stored, x_rows, noise_delta);
  if (MECH != kNoMask || x_rows != rows) return SPL_ESHAPE;
  return launch_pdl(split_fp16_kernel, grid, block, 0, stream, hi, lo, row_exp, src, cols);
}

spl_status run_split_fp16(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* src, int64_t rows, int64_t cols,
                          cudaStream_t stream) {
  if (rows == 0) return SPL_OK;
  if (rows > 0x7fffffffLL) return SPL_ESHAPE;
  return launch_split_rows<kNoMask>(hi, lo, row_exp, src, rows, cols, nullptr, 0.f, spl_rng{}, stream);
}

spl_status run_split_tf32(float* hi, float* lo, const float* src, int64_t count, cudaStream_t stream) {
  if (count == 0) return SPL_OK;
  return launch_pdl(split_tf32_kernel, dim3(grid_for(ceil_div(count, 4), 8)), dim3(kThreads), 0, stream, hi, lo, src,
                    count);
}

spl_status run_addsub(float* out, const float* a, const float* b, int64_t n, bool sub, cudaStream_t stream) {
  if (n == 0) return SPL_OK;
  const int grid = grid_for(ceil_div(n, 4), 8);
  if (sub) {
    addsub_kernel<true><<<grid, kThreads, 0, stream>>>(out, a, b, n);
  } else {
    addsub_kernel<false><<<grid, kThreads, 0, stream>>>(out, a, b, n);
  }
  return launch_status();
}

}  // namespace spl

using namespace spl;

extern "C" spl_status spl_noise(float* N, int64_t rows, int64_t cols, double sensitivity, double eps, spl_mech mech,
                                spl_rng rng, cudaStream_t stream) {
  spl_status st = validate_noise(rows, cols, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  const int64_t n = rows * cols;
  if (n == 0) return SPL_OK;
  if (!N) return SPL_EINVAL;
  if (!aligned16(N)) return SPL_EALIGN;
  return launch_noise_mask(nullptr, N, nullptr, n, sensitivity, eps, mech, rng, stream);
}

extern "C" spl_status spl_random_bits(uint32_t* out, int64_t count, spl_rng rng, cudaStream_t stream) {
  if (count < 0) return SPL_EINVAL;
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  if (count == 0) return SPL_OK;
  if (!out) return SPL_EINVAL;
  if (!aligned16(out)) return SPL_EALIGN;
  return launch_pdl(random_bits_kernel, dim3(grid_for(ceil_div(count, 4), 8)), dim3(kThreads), 0, stream, out, count,
                    make_philox_key(rng.seed, rng.stream_id), rng.offset, rng.offset_dev);
}

extern "C" spl_status spl_rng_advance(uint64_t* offset_dev, uint64_t delta, cudaStream_t stream) {
  if (!offset_dev) return SPL_EINVAL;
  if ((reinterpret_cast<uintptr_t>(offset_dev) & 7u) != 0) return SPL_EALIGN;
  return launch_pdl(rng_advance_kernel, dim3(1), dim3(1), 0, stream, offset_dev, delta);
}

extern "C" spl_status spl_noise_mask(float* Xt, float* N_out, const float* X, int64_t rows, int64_t cols,
                                     double sensitivity, double eps, spl_mech mech, spl_rng rng,
                                     cudaStream_t stream) {
  spl_status st = validate_noise(rows, cols, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  const int64_t n = rows * cols;
  if (n == 0) return SPL_OK;
  if (!Xt || !X) return SPL_EINVAL;
  if (!aligned16(Xt) || !aligned16(X) || (N_out && !aligned16(N_out))) return SPL_EALIGN;
  return launch_noise_mask(Xt, N_out, X, n, sensitivity, eps, mech, rng, stream);
}

extern "C" spl_status spl_noise_mask_f64(double* Xt, const float* X, int64_t rows, int64_t cols, double sensitivity,
                                         double eps, spl_mech mech, spl_rng rng, cudaStream_t stream) {
  spl_status st = validate_noise(rows, cols, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  const int64_t n = rows * cols;
  if (n == 0) return SPL_OK;
  if (!Xt || !X) return SPL_EINVAL;
  if (!aligned16(Xt) || !aligned16(X)) return SPL_EALIGN;
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  const float b = std::isinf(eps) ? 0.0f : (float)(sensitivity / eps);
  const int grid = grid_for(ceil_div(n, 4), 8);
  const PhiloxKey key = make_philox_key(rng.seed, rng.stream_id);
  if (b == 0.0f)
    return launch_pdl(noise_mask_f64_kernel<kZero>, dim3(grid), dim3(kThreads), 0, stream, Xt, X, n, b, key, rng.offset, rng.offset_dev);
  if (mech == SPL_MECH_LAPLACE)
    return launch_pdl(noise_mask_f64_kernel<kLaplace>, dim3(grid), dim3(kThreads), 0, stream, Xt, X, n, b, key, rng.offset, rng.offset_dev);
  return launch_pdl(noise_mask_f64_kernel<kGaussian>, dim3(grid), dim3(kThreads), 0, stream, Xt, X, n, b, key, rng.offset, rng.offset_dev);
}

extern "C" spl_status spl_slalom_mask(float* Xt, float* eta, const float* X, int64_t rows, int64_t cols, spl_rng rng,
                                      cudaStream_t stream) {
  if (rows < 0 || cols < 0) return SPL_EINVAL;
  const int64_t n = rows * cols;
  if (n == 0) return SPL_OK;
  if (!Xt || !X) return SPL_EINVAL;
  if (rng.offset_dev) return SPL_EINVAL;  // host offsets only
  const int grid = grid_for(ceil_div(n, 2), 8);
  return launch_pdl(slalom_mask_kernel, dim3(grid), dim3(kThreads), 0, stream, Xt, eta, X, n,
                    make_philox_key(rng.seed, rng.stream_id), rng.offset);
}

extern "C" spl_status spl_slalom_quantize(float* out, const float* v, int64_t count, cudaStream_t stream) {
  if (count < 0) return SPL_EINVAL;
  if (count == 0) return SPL_OK;
  if (!out || !v) return SPL_EINVAL;
  return launch_pdl(slalom_quantize_kernel, dim3(grid_for(count, 8)), dim3(kThreads), 0, stream, out, v, count);
}

extern "C" spl_status spl_noise_mask_split(float* Xt, uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* X,
                                           int64_t rows, int64_t cols, double sensitivity, double eps, spl_mech mech,
                                           spl_rng rng, cudaStream_t stream) {
  spl_status st = validate_noise(rows, cols, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  if (rows == 0 || cols == 0) return SPL_OK;
  if (!hi || !lo || !row_exp) return SPL_EINVAL;  // X NULL: the split of the noise itself
  if ((cols & 7) != 0) return SPL_EALIGN;
  if ((X && !aligned16(X)) || !aligned16(hi) || !aligned16(lo) || (Xt && !aligned16(Xt))) return SPL_EALIGN;
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  if (rows > 0x7fffffffLL) return SPL_ESHAPE;
  const float b = std::isinf(eps) ? 0.0f : (float)(sensitivity / eps);
  if (b == 0.0f) return launch_split_rows<kZero>(hi, lo, row_exp, X, rows, cols, Xt, b, rng, stream);
  if (mech == SPL_MECH_LAPLACE) return launch_split_rows<kLaplace>(hi, lo, row_exp, X, rows, cols, Xt, b, rng, stream);
  return launch_split_rows<kGaussian>(hi, lo, row_exp, X, rows, cols, Xt, b, rng, stream);
}

extern "C" spl_status spl_noise_mask_split_stacked(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* X,
                                                   int64_t x_rows, int64_t noise_rows, int64_t cols,
                                                   double sensitivity, double eps, spl_mech mech, spl_rng rng,
                                                   uint64_t noise_block_delta, cudaStream_t stream) {
  spl_status st = validate_noise(x_rows, cols, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  if (noise_rows < 0) return SPL_EINVAL;
  const int64_t rows = x_rows + noise_rows;
  if (rows == 0 || cols == 0) return SPL_OK;
  if (!hi || !lo || !row_exp || (x_rows > 0 && !X)) return SPL_EINVAL;
  if ((cols & 7) != 0) return SPL_EALIGN;
  if ((X && !aligned16(X)) || !aligned16(hi) || !aligned16(lo)) return SPL_EALIGN;
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  if (rows > 0x7fffffffLL) return SPL_ESHAPE;
  const float b = std::isinf(eps) ? 0.0f : (float)(sensitivity / eps);
  if (b == 0.0f)
    return launch_split_rows<kZero>(hi, lo, row_exp, X, rows, cols, nullptr, b, rng, stream, nullptr, x_rows,
                                    noise_block_delta);
  if (mech == SPL_MECH_LAPLACE)
    return launch_split_rows<kLaplace>(hi, lo, row_exp, X, rows, cols, nullptr, b, rng, stream, nullptr, x_rows,
                                       noise_block_delta);
  return launch_split_rows<kGaussian>(hi, lo, row_exp, X, rows, cols, nullptr, b, rng, stream, nullptr, x_rows,
                                      noise_block_delta);
}

extern "C" spl_status spl_mask_split(float* Xt, uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* X,
                                     const float* N, int64_t rows, int64_t cols, cudaStream_t stream) {
  if (rows < 0 || cols < 0) return SPL_EINVAL;
  if (rows == 0 || cols == 0) return SPL_OK;
  if (!hi || !lo || !row_exp || !X || !N) return SPL_EINVAL;
  if ((cols & 7) != 0) return SPL_EALIGN;
  if (!aligned16(X) || !aligned16(N) || !aligned16(hi) || !aligned16(lo) || (Xt && !aligned16(Xt))) return SPL_EALIGN;
  if (rows > 0x7fffffffLL) return SPL_ESHAPE;
  return launch_split_rows<kStored>(hi, lo, row_exp, X, rows, cols, Xt, 0.0f, spl_rng{}, stream, N);
}

extern "C" spl_status spl_mask(float* Xt, const float* X, const float* N, int64_t rows, int64_t cols,
                               cudaStream_t stream) {
  if (rows < 0 || cols < 0) return SPL_EINVAL;
  const int64_t n = rows * cols;
  if (n == 0) return SPL_OK;
  if (!Xt || !X || !N) return SPL_EINVAL;
  if (!aligned16(Xt) || !aligned16(X) || !aligned16(N)) return SPL_EALIGN;
  return run_addsub(Xt, X, N, n, false, stream);
}

extern "C" spl_status spl_unmask(float* Y, const float* Yt, const float* C, int64_t rows, int64_t cols,
                                 cudaStream_t stream) {
  if (rows < 0 || cols < 0) return SPL_EINVAL;
  const int64_t n = rows * cols;
  if (n == 0) return SPL_OK;
  if (!Y || !Yt || !C) return SPL_EINVAL;
  if (!aligned16(Y) || !aligned16(Yt) || !aligned16(C)) return SPL_EALIGN;
  return run_addsub(Y, Yt, C, n, true, stream);
}

extern "C" spl_status spl_split_fp16(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* src, int64_t rows,
                                     int64_t cols, cudaStream_t stream) {
  if (rows < 0 || cols < 0) return SPL_EINVAL;
  if (rows == 0) return SPL_OK;
  if (!row_exp || (cols > 0 && (!hi || !lo || !src))) return SPL_EINVAL;
  if ((cols & 7) != 0) return SPL_EALIGN;
  if ((hi && !aligned16(hi)) || (lo && !aligned16(lo)) || (src && !aligned16(src))) return SPL_EALIGN;
  if (cols == 0) return cudaMemsetAsync(row_exp, 0, (size_t)rows * sizeof(int32_t), stream) == cudaSuccess
                            ? SPL_OK : SPL_ECUDA;
  return run_split_fp16(hi, lo, row_exp, src, rows, cols, stream);
}

extern "C" spl_status spl_split_tf32(float* hi, float* lo, const float* src, int64_t count, cudaStream_t stream) {
  if (count < 0) return SPL_EINVAL;
  if (count == 0) return SPL_OK;
  if (!hi || !lo || !src) return SPL_EINVAL;
  if (!aligned16(hi) || !aligned16(lo) || !aligned16(src)) return SPL_EALIGN;
  return run_split_tf32(hi, lo, src, count, stream);
}

// The boundary's listed name for the TF32X3 weight split: spl_split_tf32 over the N x K weight.
extern "C" spl_status spl_prepare_weight_split(float* W_hi, float* W_lo, const float* W, int64_t N, int64_t K,
                                               cudaStream_t stream) {
  if (N < 0 || K < 0) return SPL_EINVAL;
  if (N > 0 && K > (int64_t(1) << 62) / N) return SPL_ESHAPE;
  return spl_split_tf32(W_hi, W_lo, W, N * K, stream);
}
