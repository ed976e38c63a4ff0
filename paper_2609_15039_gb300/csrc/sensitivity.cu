// a1: noise scale inputs.  Global l2 sensitivities of the functions that feed
// each offloaded projection (Sec. 4.3, Thms. 1-3), evaluated in fp64 on the
// host, and the spectral norm ||W||_2 (Eq. matrix-norm) of a device matrix by
// power iteration on W^T W.
//
// Dimension reading for Thm. 3 (Sec. 4.3 says to use the dimension of each
// operation): the leading sqrt(d) bounds ||sig(g(x))||_2 with g(x) in R^{d_ff},
// so it is sqrt(d_ff); the LN factor uses the model dimension d.

#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace spl {
namespace {

double norm4_host(const float* a, int64_t d) {
  long double s = 0.0L;
  for (int64_t i = 0; i < d; ++i) {
    const long double v = (long double)a[i];
    s += v * v * v * v;
  }
  return (double)std::pow((double)s, 0.25);
}

// Deterministic start vector in [-1, 1] (integer hash of the index).
__device__ __forceinline__ float start_value(int64_t k) {
  uint32_t h = (uint32_t)k * 0x9E3779B1u + 0x7F4A7C15u;
  h ^= h >> 15;
  h *= 0x2C1B3C6Du;
  h ^= h >> 12;
  h *= 0x297A2D39u;
  h ^= h >> 15;
  return (float)(h >> 8) * (2.0f / 16777216.0f) - 1.0f;
}

__global__ void init_v_kernel(float* v, int64_t K) {
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K; k += (int64_t)gridDim.x * blockDim.x)
    v[k] = start_value(k);
}

// u = W v, one warp per row.
__global__ void matvec_kernel(float* __restrict__ u, const float* __restrict__ W, const float* __restrict__ v,
                              int64_t N, int64_t K) {
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= N) return;
  const float* w = W + warp * K;
  float s = 0.f;
  for (int64_t k = lane; k < K; k += 32) s = fmaf(w[k], v[k], s);
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) u[warp] = s;
}

// vt += W[n0:n1]^T u[n0:n1] for a block of 256 columns and a range of rows.
__global__ void matvec_t_kernel(float* __restrict__ vt, const float* __restrict__ W, const float* __restrict__ u,
                                int64_t N, int64_t K, int64_t rows_per_block) {
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t n0 = (int64_t)blockIdx.y * rows_per_block;
  const int64_t n1 = n0 + rows_per_block < N ? n0 + rows_per_block : N;
  if (k >= K) return;
  float s = 0.f;
  for (int64_t n = n0; n < n1; ++n) s = fmaf(W[n * K + k], u[n], s);
  atomicAdd(vt + k, s);
}

// *nrm = ||x||_2 (fp64).  Single block.
__global__ void norm_kernel(double* nrm, const float* x, int64_t n) {
  __shared__ double red[32];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < n; i += blockDim.x) s += (double)x[i] * (double)x[i];
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    s = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0;
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (threadIdx.x == 0) *nrm = sqrt(s);
  }
}

// v = vt / ||vt||, vt = 0
__global__ void rescale_kernel(float* v, float* vt, const double* nrm, int64_t K) {
  const double n = *nrm;
  const float inv = n > 0.0 ? (float)(1.0 / n) : 0.0f;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K; k += (int64_t)gridDim.x * blockDim.x) {
    v[k] = vt[k] * inv;
    vt[k] = 0.f;
  }
}

}  // namespace
}  // namespace spl

using namespace spl;

extern "C" double spl_delta_layernorm(const float* alpha, int64_t d) {
  if (!alpha || d <= 0) return -1.0;
  return 2.0 * std::sqrt((double)d) * norm4_host(alpha, d);
}

extern "C" double spl_delta_attention(const float* alpha, int64_t d, double wval_spectral_norm) {
  if (!alpha || d <= 0 || !(wval_spectral_norm >= 0.0)) return -1.0;
  return 2.0 * std::sqrt((double)d) * wval_spectral_norm * norm4_host(alpha, d);
}

extern "C" double spl_delta_activation(const float* alpha, const float* beta, int64_t d, int64_t d_ff,
                                       double wup_spectral_norm, double wgate_spectral_norm) {
  if (!alpha || d <= 0 || d_ff <= 0 || !(wup_spectral_norm >= 0.0) || !(wgate_spectral_norm >= 0.0)) return -1.0;
  long double b2 = 0.0L;
  if (beta)
    for (int64_t i = 0; i < d; ++i) b2 += (long double)beta[i] * (long double)beta[i];
  const double ln_bound = std::sqrt((double)d) * norm4_host(alpha, d) + std::sqrt((double)b2);
  return 2.0 * std::sqrt((double)d_ff) * ln_bound * ln_bound * wup_spectral_norm * wgate_spectral_norm;
}

extern "C" spl_status spl_spectral_norm(double* out, const float* W, int64_t N, int64_t K, int iters,
                                        void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  if (!out || !W || N <= 0 || K <= 0 || iters < 1) return SPL_EINVAL;
  const size_t need = (size_t)4 * (size_t)(N + 2 * K) + 256;
  if (!workspace || workspace_bytes < need) return SPL_EWORKSPACE;
  if (!aligned16(W) || !aligned16(workspace)) return SPL_EALIGN;
  char* ws = static_cast<char*>(workspace);
  double* nrm = reinterpret_cast<double*>(ws);
  float* u = reinterpret_cast<float*>(ws + 256);
  float* v = u + N;
  float* vt = v + K;
  const int sms = device_sm_count();
  const int ew_grid = (int)std::min<int64_t>(ceil_div(K, 256), (int64_t)sms * 4);
  init_v_kernel<<<ew_grid, 256, 0, stream>>>(v, K);
  if (cudaMemsetAsync(vt, 0, (size_t)K * 4, stream) != cudaSuccess) return SPL_ECUDA;
  const int64_t rows_per_block = std::max<int64_t>(64, ceil_div(N, 64));
  const dim3 tgrid((unsigned)ceil_div(K, 256), (unsigned)ceil_div(N, rows_per_block));
  const unsigned mv_grid = (unsigned)ceil_div(N * 32, 256);
  for (int it = 0; it < iters; ++it) {
    matvec_kernel<<<mv_grid, 256, 0, stream>>>(u, W, v, N, K);
    matvec_t_kernel<<<tgrid, 256, 0, stream>>>(vt, W, u, N, K, rows_per_block);
    norm_kernel<<<1, 1024, 0, stream>>>(nrm, vt, K);
    rescale_kernel<<<ew_grid, 256, 0, stream>>>(v, vt, nrm, K);
  }
  matvec_kernel<<<mv_grid, 256, 0, stream>>>(u, W, v, N, K);
  norm_kernel<<<1, 1024, 0, stream>>>(nrm, u, N);
  note_launches(3 + 4 * (uint64_t)iters);
  if (cudaGetLastError() != cudaSuccess) return SPL_ECUDA;
  if (cudaMemcpyAsync(out, nrm, sizeof(double), cudaMemcpyDeviceToHost, stream) != cudaSuccess) return SPL_ECUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return SPL_ECUDA;
  return SPL_OK;
}
