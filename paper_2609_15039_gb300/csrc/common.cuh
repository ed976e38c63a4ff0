// Internal helpers shared by the library's translation units.
#pragma once

#include <cstdint>
#include <cmath>

#include <cuda_runtime.h>

#include "spl.h"

namespace spl {

constexpr int kNumSMsGB300 = 152;

// Device status word: bit set by kernels whose bounded waits expired.  It lives
// in the translation unit of the only kernels that wait (gemm_tc.cu); this
// reads it and clears it (synchronously).
constexpr unsigned int kStatusTimeout = 1u;
cudaError_t read_clear_device_status(unsigned int* word);

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Running count of kernels this library has launched (spl_launch_count).
void note_launches(uint64_t n);

// Call once right after each kernel launch: counts it and maps the launch error.
inline spl_status launch_status() {
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
}

// Number of SMs of the current device (cached per device).
int device_sm_count();
// Compute capability major*10+minor of the current device.
int device_cc();

// ---- product dispatch shared by gemm_simt.cu, gemv.cu, gemm_tc.cu, linear.cu ----
struct LinearArgs {
  float* out;            // [M, N]
  const float* a;        // [M, K]  (X~ or noise)
  const float* w;        // [N, K]
  const float* w_hi;     // [N, K] or null
  const float* w_lo;     // [N, K] or null
  const float* c;        // [M, N] correction subtracted in the epilogue, or null
  int64_t M, K, N;
  void* ws;              // workspace (zero-filled), may be null
  size_t ws_bytes;
  cudaStream_t stream;
};

// Workspace layout shared by every product call: the first kCounterBytes hold
// the decode kernel's arrival counters (zero between calls); split-K partials
// and the TF32 split of the left operand follow.  Keeping the counters at a
// fixed place lets one workspace serve calls of any shape and path.
constexpr size_t kCounterBytes = 64 * 1024;
constexpr int64_t kMaxCounters = (int64_t)(kCounterBytes / sizeof(unsigned int));

// Split-K plans: how many K-splits each kernel uses and the workspace it needs.
struct Plan {
  int kernel;            // 0 = GEMV (decode), 1 = FP32 SIMT GEMM, 2 = TF32X3 tcgen05 GEMM
  int splits;            // K-splits (1 = none)
  int64_t k_per_split;   // multiple of the kernel's K granule
  size_t ws_partials;    // bytes of split partials (at offset kCounterBytes)
  size_t ws_asplit;      // bytes of the A operand's hi/lo split (TF32X3, after the partials)
  size_t total() const { return (ws_partials + ws_asplit) ? kCounterBytes + ws_partials + ws_asplit : 0; }
};

constexpr int kGemvMaxM = 16;
constexpr int kKernelGemv = 0, kKernelSimt = 1, kKernelTc = 2;

Plan plan_gemv(int64_t M, int64_t K, int64_t N, int sms);
Plan plan_simt(int64_t M, int64_t K, int64_t N, int sms);
Plan plan_tc(int64_t M, int64_t K, int64_t N, int sms);

spl_status run_gemv(const LinearArgs& a, const Plan& p);
int64_t gemv_max_ks(int64_t M);                           // largest K-slice the decode kernel stages for M rows
int tc_uniform_splits(int64_t M, int64_t K, int64_t N);    // K-split of a one-launch TF32X3 call, 0 if mixed
spl_status run_tc_splits(const LinearArgs& a, int splits); // TF32X3 with the same K-split on every tile
spl_status run_simt(const LinearArgs& a, const Plan& p);
spl_status run_tc(const LinearArgs& a, const Plan& p);

// Deterministic split-K reduction: out = sum_s part[s] (in s order) - c.
spl_status run_splitk_reduce(float* out, const float* part, const float* c, int splits, int64_t M,
                             int64_t N, cudaStream_t stream);

// Elementwise TF32 split (used for the A operand of TF32X3 inside the workspace).
spl_status run_split_tf32(float* hi, float* lo, const float* src, int64_t count, cudaStream_t stream);

__host__ __device__ inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
__host__ __device__ inline int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

}  // namespace spl
