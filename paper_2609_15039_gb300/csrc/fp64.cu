// The binary64 path of Sec. 5.5 ("The Case Against the Down Linear Projection"): the input of Down
// is masked with noise whose scale follows the activation bound of Thm. 3, so large that in
// binary32 the cancellation error of Eq. fp-log-bound (u = 2^-24) swamps the output.  In binary64
// (p = 53) gamma_d shrinks by 2^29 and the recovered output is accurate again.  Here the whole
// computation is binary64: the mask is rounded once in binary64 (spl_noise_mask_f64), every
// product of the masked input and the fp32 weight is rounded once in binary64 and summed in
// binary64, the correction W eta is kept in binary64 and subtracted in binary64; only Y is rounded
// to fp32 at the end.
//
// Kernel: the decode kernel's structure in binary64 -- a 256-thread block owns 16 rows of W over
// a K-slice, stages MT (1, 2, 4 or 8) rows of the left operand of that slice in shared memory (as
// binary64), streams W once and keeps 2 x MT binary64 partial sums per lane, reduced across the
// warp; a grid dimension walks MT-row chunks of the left operand.  K-split partials go to the workspace
// (binary64) and a second kernel sums them in split order and writes C or Y = fl32(r - C).
// Bound by the FP64 rate (2 M K N flops at the DFMA peak), not by HBM.

#include <algorithm>

#include "common.cuh"

namespace spl {
namespace {

constexpr int THREADS = 256, WARPS = 8, ROWS = 2;  // rows of W per warp
constexpr int SMEM_DOUBLES = 6144;                  // 48 KB of staged A
// rows of A per block: 1, 2, 4 or 8 (the smallest that covers M, 8 beyond)
inline int mt_for(int64_t M) { return M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : 8; }
inline int64_t max_ks(int mt) { return SMEM_DOUBLES / mt / 128 * 128; }

template <typename TA>
__device__ __forceinline__ double2 load_a2(const TA* p);
template <>
__device__ __forceinline__ double2 load_a2<float>(const float* p) {
  const float2 v = __ldg(reinterpret_cast<const float2*>(p));
  return make_double2((double)v.x, (double)v.y);
}
template <>
__device__ __forceinline__ double2 load_a2<double>(const double* p) {
  return __ldg(reinterpret_cast<const double2*>(p));
}

// Final value of an output (one split, or after the split-order reduction):
//   kOut64  out64 = acc (the correction C, binary64)
//   kUnmask out32 = fl32(acc - c)
//   kSlalom out32 = ((acc - c) mod q, taken in (-q/2, q/2]) 2^-16: the Slalom comparator's unmask
//           and de-quantization (Sec. 6.2); acc and c are exact integers in binary64.
enum { kOut64 = 0, kUnmask = 1, kSlalom = 2 };
constexpr double kSlalomQ = 10485767.0;  // 2^23 + 2^21 + 7

__device__ __forceinline__ void finish(double* out64, float* out32, int64_t o, double acc, const double* c, int mode) {
  if (mode == kOut64) {
    out64[o] = acc;
  } else if (mode == kUnmask) {
    out32[o] = (float)(acc - c[o]);
  } else {
    const double t = acc - c[o];  // exact integer, |t| < 2^53
    double m = t - kSlalomQ * floor(t / kSlalomQ);
    if (m < 0.0) m += kSlalomQ;
    if (m >= kSlalomQ) m -= kSlalomQ;
    if (m > (kSlalomQ - 1.0) * 0.5) m -= kSlalomQ;
    out32[o] = (float)(m * 0x1p-16);
  }
}

// part[split][m][n] (splits > 1) or, with one split, the final value (see finish).
template <typename TA, int MT>
__global__ void __launch_bounds__(THREADS) gemv_f64_kernel(double* __restrict__ out64, float* __restrict__ out32,
                                                           const TA* __restrict__ A, const float* __restrict__ W,
                                                           const double* __restrict__ c, int64_t M, int64_t K,
                                                           int64_t N, int64_t ks, int splits, int mode) {
  extern __shared__ __align__(16) double as[];  // [MT][ks]
  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.y;
  const int64_t mbase = (int64_t)blockIdx.z * MT;
  const int64_t k0 = (int64_t)split * ks;
  const int64_t klen = std::min<int64_t>(ks, K - k0);  // multiple of 4 (or <= 0: empty split)
  const int64_t q2 = klen > 0 ? klen >> 1 : 0;
  for (int64_t q = threadIdx.x; q < (int64_t)MT * q2; q += THREADS) {
    const int m = (int)(q / q2);
    const int64_t k = (q - (int64_t)m * q2) * 2;
    double2 v = make_double2(0.0, 0.0);
    if (mbase + m < M) v = load_a2<TA>(A + (mbase + m) * K + k0 + k);
    *reinterpret_cast<double2*>(as + (int64_t)m * ks + k) = v;
  }
  __syncthreads();
  const int64_t nbase = (int64_t)blockIdx.x * (WARPS * ROWS) + warp * ROWS;
  double acc[ROWS][MT];
#pragma unroll
  for (int r = 0; r < ROWS; ++r)
#pragma unroll
    for (int m = 0; m < MT; ++m) acc[r][m] = 0.0;
  for (int64_t kk = lane * 4; kk < klen; kk += 128) {
    float4 wv[ROWS];
#pragma unroll
    for (int r = 0; r < ROWS; ++r)
      wv[r] = nbase + r < N ? __ldcs(reinterpret_cast<const float4*>(W + (nbase + r) * K + k0 + kk))
                            : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      const double2 x01 = *reinterpret_cast<const double2*>(as + (int64_t)m * ks + kk);
      const double2 x23 = *reinterpret_cast<const double2*>(as + (int64_t)m * ks + kk + 2);
#pragma unroll
      for (int r = 0; r < ROWS; ++r) {
        double a = acc[r][m];
        a = fma(x01.x, (double)wv[r].x, a);
        a = fma(x01.y, (double)wv[r].y, a);
        a = fma(x23.x, (double)wv[r].z, a);
        a = fma(x23.y, (double)wv[r].w, a);
        acc[r][m] = a;
      }
    }
  }
#pragma unroll
  for (int r = 0; r < ROWS; ++r)
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      double v = acc[r][m];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      acc[r][m] = v;
    }
  if (lane != 0) return;
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    const int64_t n = nbase + r;
    if (n >= N) continue;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      const int64_t row = mbase + m;
      if (row >= M) continue;
      const int64_t o = row * N + n;
      if (splits > 1)
        out64[(int64_t)split * M * N + o] = acc[r][m];
      else
        finish(out64, out32, o, acc[r][m], c, mode);
    }
  }
}

// Sum of the split partials in split order; then C64 (out64) or Y = fl32(sum - c) (out32).
__global__ void __launch_bounds__(256) reduce_f64_kernel(double* __restrict__ out64, float* __restrict__ out32,
                                                         const double* __restrict__ part, const double* __restrict__ c,
                                                         int splits, int64_t total, int mode) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    double s = part[i];
    for (int sp = 1; sp < splits; ++sp) s += part[(int64_t)sp * total + i];
    finish(out64, out32, i, s, c, mode);
  }
}

struct PlanF64 {
  int mt;
  int64_t ks;
  int splits;
  size_t ws;
};

PlanF64 plan_f64(int64_t M, int64_t K, int64_t N) {
  PlanF64 p;
  p.mt = mt_for(M);
  const int64_t groups = ceil_div(N, WARPS * ROWS) * ceil_div(M, p.mt);
  const int64_t target = (int64_t)device_sm_count() * 4;
  int64_t s = std::max<int64_t>(ceil_div(K, max_ks(p.mt)), ceil_div(target, groups));
  s = std::min<int64_t>(s, std::max<int64_t>(1, K / 128));
  p.ks = std::min<int64_t>(round_up(ceil_div(K, s), 128), max_ks(p.mt));
  p.splits = (int)ceil_div(K, p.ks);
  // partials after the decode kernel's counter region, which must stay untouched (zero)
  p.ws = p.splits > 1 ? kCounterBytes + (size_t)round_up((int64_t)p.splits * M * N * 8, 256) : 0;
  return p;
}

template <typename TA, int MT>
spl_status launch_f64(const PlanF64& p, double* out64, float* out32, const TA* A, const float* W, const double* c,
                      int64_t M, int64_t K, int64_t N, void* ws, cudaStream_t stream, int mode) {
  const dim3 grid((unsigned)ceil_div(N, WARPS * ROWS), (unsigned)p.splits, (unsigned)ceil_div(M, MT));
  if (grid.y > 65535u || grid.z > 65535u) return SPL_ESHAPE;
  const size_t smem = (size_t)MT * p.ks * sizeof(double);
  if (p.splits == 1)
    return launch_pdl(gemv_f64_kernel<TA, MT>, grid, dim3(THREADS), smem, stream, out64, out32, A, W, c, M, K, N, p.ks,
                      1, mode);
  double* part = reinterpret_cast<double*>(static_cast<char*>(ws) + kCounterBytes);
  spl_status st = launch_pdl(gemv_f64_kernel<TA, MT>, grid, dim3(THREADS), smem, stream, part, (float*)nullptr, A, W,
                             (const double*)nullptr, M, K, N, p.ks, p.splits, (int)kOut64);
  if (st != SPL_OK) return st;
  const int64_t total = M * N;
  const int rgrid = (int)std::max<int64_t>(1, std::min<int64_t>(ceil_div(total, 256), (int64_t)device_sm_count() * 8));
  return launch_pdl(reduce_f64_kernel, dim3(rgrid), dim3(256), 0, stream, out64, out32, (const double*)part, c,
                    p.splits, total, mode);
}

template <typename TA>
spl_status run_f64(double* out64, float* out32, const TA* A, const float* W, const double* c, int64_t M, int64_t K,
                   int64_t N, void* ws, size_t ws_bytes, cudaStream_t stream, int mode) {
  if (M < 0 || K < 0 || N < 0) return SPL_EINVAL;
  if (M == 0 || N == 0) return SPL_OK;
  if ((!out64 && !out32) || (out32 && !c) || (K > 0 && (!A || !W))) return SPL_EINVAL;
  if ((K & 3) != 0) return SPL_EALIGN;
  if ((A && !aligned16(A)) || (W && !aligned16(W)) || (c && !aligned16(c)) || (out64 && !aligned16(out64)) ||
      (out32 && !aligned16(out32)))
    return SPL_EALIGN;
  if (M > 0x7fffffffLL || N > 0x7fffffffLL || K > 0x7fffffffLL) return SPL_ESHAPE;
  const PlanF64 p = plan_f64(M, K, N);
  if (p.ws > 0 && (!ws || ws_bytes < p.ws)) return SPL_EWORKSPACE;
  if (ws && !aligned16(ws)) return SPL_EALIGN;
  switch (p.mt) {
    case 1: return launch_f64<TA, 1>(p, out64, out32, A, W, c, M, K, N, ws, stream, mode);
    case 2: return launch_f64<TA, 2>(p, out64, out32, A, W, c, M, K, N, ws, stream, mode);
    case 4: return launch_f64<TA, 4>(p, out64, out32, A, W, c, M, K, N, ws, stream, mode);
    default: return launch_f64<TA, 8>(p, out64, out32, A, W, c, M, K, N, ws, stream, mode);
  }
}

}  // namespace
}  // namespace spl

using namespace spl;

extern "C" size_t spl_f64_workspace_bytes(int64_t M, int64_t K, int64_t N) {
  if (M <= 0 || K <= 0 || N <= 0) return 0;
  return plan_f64(M, K, N).ws;
}

extern "C" spl_status spl_precompute_noise_product_f64(double* C, const float* Nz, const float* W, int64_t M,
                                                       int64_t K, int64_t N, void* workspace, size_t workspace_bytes,
                                                       cudaStream_t stream) {
  return run_f64<float>(C, nullptr, Nz, W, nullptr, M, K, N, workspace, workspace_bytes, stream, kOut64);
}

extern "C" spl_status spl_masked_linear_unmask_f64(float* Y, const double* Xt, const float* W, const double* C,
                                                   int64_t M, int64_t K, int64_t N, void* workspace,
                                                   size_t workspace_bytes, cudaStream_t stream) {
  return run_f64<double>(nullptr, Y, Xt, W, C, M, K, N, workspace, workspace_bytes, stream, kUnmask);
}

extern "C" spl_status spl_slalom_linear_unmask(float* Y, const float* Xt_q, const float* W_q, const double* C,
                                               int64_t M, int64_t K, int64_t N, void* workspace, size_t workspace_bytes,
                                               cudaStream_t stream) {
  if (K >= (int64_t(1) << 22)) return SPL_ESHAPE;  // keeps every integer sum below 2^53
  return run_f64<float>(nullptr, Y, Xt_q, W_q, C, M, K, N, workspace, workspace_bytes, stream, kSlalom);
}
