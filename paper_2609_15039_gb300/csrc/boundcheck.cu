// a8: the paper's cancellation bound evaluated on the GPU, and the path choice built on it.
//
// Sec. 4.5 proves the bound of Thm. 4 and proposes Eq. fp-log-bound as a closer estimate;
// the paper uses them to judge, from sampled inputs and masks alone, whether the error of a
// configuration is acceptable (Sec. 4.5, Sec. 6.3.2).  spl_bound_check does that on the GPU:
// for a block of rows it computes, in fp64 (products of fp32 values are exact in fp64),
// the exact product Y* = X W^T and the three sums S_x = <|w|,|x|>, S_xt = <|w|,|x~|>,
// S_n = <|w|,|eta|>, then compares the recovered output Y with
//   hard = gamma_K (S_x + S_xt + S_n) + u S_x + u S_xt (1+u)/(1-u) + u gamma_K (S_x + S_xt + S_n)
//          (Thm. 4 with the rounding of the mask and the second-order term written out)
//   log  = gamma_{ceil(log2 K)+1} (S_x + S_xt + S_n) + u S_x          (Eq. fp-log-bound)
// with u = 2^-24 and gamma_n = n u / (1 - n u) (Def. u-and-theta).
//
// spl_choose_path masks a sample, runs the correction and the masked product with each path
// (FP32, TF32X3, FP16X3), checks each against the bound and picks a tensor-core path only
// when it stays inside the hard bound and its log-bound violations and mean error are no
// worse than FP32's; FP16X3 is tried first.

#include <algorithm>
#include <cmath>
#include <cstring>

#include "common.cuh"

namespace spl {
namespace {

enum { kMaxErrHard = 0, kMaxErrLog, kViolLog, kSumErr, kSumLog, kSumHard, kCount, kMaxRef, kMaxErr, kNumStats };

__device__ __forceinline__ void atomic_max_nonneg(double* addr, double v) {
  // non-negative doubles order like their bit patterns
  atomicMax(reinterpret_cast<unsigned long long*>(addr), (unsigned long long)__double_as_longlong(v));
}

// One warp per output (r, n): lanes stride over K with fp64 accumulators.
__global__ void __launch_bounds__(256) bound_check_kernel(double* __restrict__ stats, const float* __restrict__ Y,
                                                          const float* __restrict__ X, const float* __restrict__ Xt,
                                                          const float* __restrict__ Nz, const float* __restrict__ W,
                                                          int64_t rows, int64_t K, int64_t N, double g_hard,
                                                          double g_log, double u) {
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows * N) return;
  const int64_t r = warp / N, n = warp % N;
  const float* x = X + r * K;
  const float* xt = Xt + r * K;
  const float* eta = Nz + r * K;
  const float* w = W + n * K;
  double ref = 0.0, sx = 0.0, sxt = 0.0, sn = 0.0;
  for (int64_t k = lane; k < K; k += 32) {
    const double wk = (double)w[k], aw = fabs(wk);
    const double xk = (double)x[k];
    ref = fma(xk, wk, ref);
    sx = fma(fabs(xk), aw, sx);
    sxt = fma(fabs((double)xt[k]), aw, sxt);
    sn = fma(fabs((double)eta[k]), aw, sn);
  }
  for (int o = 16; o > 0; o >>= 1) {
    ref += __shfl_xor_sync(0xffffffffu, ref, o);
    sx += __shfl_xor_sync(0xffffffffu, sx, o);
    sxt += __shfl_xor_sync(0xffffffffu, sxt, o);
    sn += __shfl_xor_sync(0xffffffffu, sn, o);
  }
  if (lane != 0) return;
  const double s3 = sx + sxt + sn;
  const double hard = g_hard * s3 + u * sx + u * sxt * (1.0 + u) / (1.0 - u) + u * g_hard * s3;
  const double logb = g_log * s3 + u * sx;
  const double err = fabs((double)Y[r * N + n] - ref);
  atomic_max_nonneg(stats + kMaxErrHard, hard > 0.0 ? err / hard : (err > 0.0 ? INFINITY : 0.0));
  atomic_max_nonneg(stats + kMaxErrLog, logb > 0.0 ? err / logb : (err > 0.0 ? INFINITY : 0.0));
  if (err > logb) atomicAdd(stats + kViolLog, 1.0);
  atomicAdd(stats + kSumErr, err);
  atomicAdd(stats + kSumLog, logb);
  atomicAdd(stats + kSumHard, hard);
  atomicAdd(stats + kCount, 1.0);
  atomic_max_nonneg(stats + kMaxRef, fabs(ref));
  atomic_max_nonneg(stats + kMaxErr, err);
}

double gamma_n(double n, double u) { return n * u / (1.0 - n * u); }

}  // namespace
}  // namespace spl

using namespace spl;

extern "C" spl_status spl_bound_check(double* stats, const float* Y, const float* X, const float* Xt, const float* Nz,
                                      const float* W, int64_t rows, int64_t K, int64_t N, void* workspace,
                                      size_t workspace_bytes, cudaStream_t stream) {
  if (!stats || rows < 0 || K < 0 || N < 0) return SPL_EINVAL;
  std::memset(stats, 0, sizeof(double) * SPL_BOUND_STATS);
  if (rows == 0 || N == 0) return SPL_OK;
  if (!Y || !X || !Xt || !Nz || !W) return SPL_EINVAL;
  if (!workspace || workspace_bytes < sizeof(double) * SPL_BOUND_STATS) return SPL_EWORKSPACE;
  const double u = std::ldexp(1.0, -24);
  const double kk = (double)std::max<int64_t>(K, 1);
  if (kk * u >= 1.0) return SPL_ESHAPE;
  const double g_hard = gamma_n(kk, u);
  const double g_log = gamma_n(std::ceil(std::log2(kk)) + 1.0, u);
  double* dstats = static_cast<double*>(workspace);
  if (cudaMemsetAsync(dstats, 0, sizeof(double) * SPL_BOUND_STATS, stream) != cudaSuccess) return SPL_ECUDA;
  const int64_t warps = rows * N;
  bound_check_kernel<<<(unsigned)ceil_div(warps * 32, 256), 256, 0, stream>>>(dstats, Y, X, Xt, Nz, W, rows, K, N,
                                                                             g_hard, g_log, u);
  spl_status st = launch_status();
  if (st != SPL_OK) return st;
  if (cudaMemcpyAsync(stats, dstats, sizeof(double) * SPL_BOUND_STATS, cudaMemcpyDeviceToHost, stream) !=
      cudaSuccess)
    return SPL_ECUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return SPL_ECUDA;
  return SPL_OK;
}

extern "C" size_t spl_choose_path_workspace_bytes(int64_t rows, int64_t K, int64_t N) {
  if (rows <= 0 || K <= 0 || N <= 0) return 0;
  const size_t f = sizeof(float);
  const size_t prod = spl_linear_workspace_bytes(rows, K, N, SPL_PATH_AUTO);  // every path
  // Xt [rows, K], C [rows, N], Y [rows, N], stats, then the product workspace
  return (size_t)round_up((int64_t)(rows * K * f), 256) + 2 * (size_t)round_up((int64_t)(rows * N * f), 256) + 256 +
         prod;
}

extern "C" spl_status spl_choose_path(spl_path* chosen, double* stats, const float* X, const float* Nz,
                                      const spl_weight* W, int64_t rows, int64_t K, int64_t N, void* workspace,
                                      size_t workspace_bytes, cudaStream_t stream) {
  if (!chosen || !stats) return SPL_EINVAL;
  *chosen = SPL_PATH_FP32;
  if (rows <= 0 || K <= 0 || N <= 0) return SPL_EINVAL;
  if (!X || !Nz || !W || !W->w) return SPL_EINVAL;
  const size_t need = spl_choose_path_workspace_bytes(rows, K, N);
  if (!workspace || workspace_bytes < need) return SPL_EWORKSPACE;
  char* ws = static_cast<char*>(workspace);
  float* xt = reinterpret_cast<float*>(ws);
  ws += round_up(rows * K * (int64_t)sizeof(float), 256);
  float* c = reinterpret_cast<float*>(ws);
  ws += round_up(rows * N * (int64_t)sizeof(float), 256);
  float* y = reinterpret_cast<float*>(ws);
  ws += round_up(rows * N * (int64_t)sizeof(float), 256);
  double* dstats = reinterpret_cast<double*>(ws);
  ws += 256;
  void* pws = ws;
  const size_t pws_bytes = workspace_bytes - (size_t)(ws - static_cast<char*>(workspace));
  spl_status st = spl_mask(xt, X, Nz, rows, K, stream);
  if (st != SPL_OK) return st;
  // stats blocks in the order FP32, TF32X3, FP16X3
  const spl_path paths[3] = {SPL_PATH_FP32, SPL_PATH_TF32X3, SPL_PATH_FP16X3};
  const int cc = device_cc();
  const bool tc = cc == 100 || cc == 103;  // tcgen05 device
  const bool have[3] = {true, tc && W->tf32_hi && W->tf32_lo,
                        tc && W->f16_hi && W->f16_lo && W->f16_exp && (K & 7) == 0};
  for (int p = 0; p < 3; ++p) {
    double* out = stats + p * SPL_BOUND_STATS;
    std::memset(out, 0, sizeof(double) * SPL_BOUND_STATS);
    out[kMaxErrHard] = INFINITY;
    if (!have[p]) continue;
    st = spl_precompute_noise_product(c, Nz, W, rows, K, N, paths[p], pws, pws_bytes, stream);
    if (st == SPL_EUNSUPPORTED && p > 0) continue;
    if (st != SPL_OK) return st;
    st = spl_masked_linear_unmask(y, xt, W, c, rows, K, N, paths[p], pws, pws_bytes, stream);
    if (st != SPL_OK) return st;
    st = spl_bound_check(out, y, X, xt, Nz, W->w, rows, K, N, dstats, 256, stream);
    if (st != SPL_OK) return st;
  }
  const double* b = stats;  // FP32
  for (int p = 2; p >= 1; --p) {  // FP16X3 first (fewer weight bytes, twice the rate), then TF32X3
    const double* a = stats + p * SPL_BOUND_STATS;
    const bool inside = a[kMaxErrHard] <= 1.0;
    const bool no_worse = a[kViolLog] <= b[kViolLog] + 0.01 * a[kCount] && a[kSumErr] <= 1.5 * b[kSumErr] + 1e-300;
    if (inside && no_worse) {
      *chosen = paths[p];
      return SPL_OK;
    }
  }
  return SPL_OK;
}
