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

// Programmatic dependent launch.  A kernel launched with launch_pdl may start while the kernel
// before it in the stream is still running; it calls pdl_wait() before it touches memory that
// kernel writes (or any memory at all, when in doubt), and pdl_trigger() once it has waited, so
// that the next kernel can be scheduled early in turn.  A dependent is scheduled only once every
// CTA of its predecessor has triggered or exited, so every CTA it could wait on has started: no
// kernel holds SM resources while waiting on one that is not yet resident, and every tensor-core
// kernel has its tensor memory before it triggers.  The fp16 split kernels therefore trigger before
// they wait: the product after a split (at most two kernels ahead) may start loading its weight
// while the kernel before the split finishes.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline spl_status launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                             Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
  note_launches(1);
  return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
}

// Number of SMs of the current device (cached per device).
int device_sm_count();
// Compute capability major*10+minor of the current device.
int device_cc();

// ---- product dispatch shared by gemm_simt.cu, gemv.cu, gemm_tc.cu, linear.cu ----
struct LinearArgs {
  float* out;               // [M, N]
  const float* a;           // [M, K]  (X~ or noise)
  const float* w;           // [N, K]  fp32
  const float* w_hi;        // [N, K]  TF32 split, or null
  const float* w_lo;
  const uint16_t* w_h16;    // [N, K]  fp16 split (binary16 bits), or null
  const uint16_t* w_l16;
  const int32_t* w_exp;     // [N]     row exponents of the fp16 split
  const float* c;           // [M, N]  correction subtracted in the epilogue, or null
  int64_t M, K, N;
  void* ws;                 // workspace (zero-filled), may be null
  size_t ws_bytes;
  cudaStream_t stream;
  spl_path path;            // resolved arithmetic path
  const uint16_t* a_h16;    // [M, K]  fp16 split of a, made by the caller (FP16X3), or null
  const uint16_t* a_l16;
  const int32_t* a_exp;     // [M]
  int64_t c_rows;           // rows of c: output rows from c_rows on subtract nothing (tensor-core and decode kernels)
};

// Workspace layout shared by every product call: the first kCounterBytes hold
// the decode kernel's arrival counters (zero between calls); split-K partials,
// or the FP16X3 split of the left operand, follow.  Keeping the counters
// at a fixed place lets one workspace serve calls of any shape and path.
constexpr size_t kCounterBytes = 64 * 1024;
constexpr int64_t kMaxCounters = (int64_t)(kCounterBytes / sizeof(unsigned int));

inline LinearArgs make_args(float* out, const float* a, const spl_weight& W, const float* c, int64_t M, int64_t K,
                            int64_t N, void* ws, size_t ws_bytes, cudaStream_t stream, spl_path path) {
  LinearArgs r{};
  r.out = out;
  r.a = a;
  r.w = W.w;
  r.w_hi = W.tf32_hi;
  r.w_lo = W.tf32_lo;
  r.w_h16 = W.f16_hi;
  r.w_l16 = W.f16_lo;
  r.w_exp = W.f16_exp;
  r.c = c;
  r.M = M;
  r.K = K;
  r.N = N;
  r.ws = ws;
  r.ws_bytes = ws_bytes;
  r.stream = stream;
  r.path = path;
  r.c_rows = M;
  return r;
}

// Power-of-two exponent e that brings max |x| of a row into [2^14, 2^15) for the fp16 split
// (0 for an all-zero row), clamped so 2^e and 2^-e stay normal floats.
__device__ __forceinline__ int fp16_row_exponent(float amax) {
  if (!(amax > 0.0f)) return 0;
  const int e = ((__float_as_int(amax) >> 23) & 0xFF) - 127;  // amax in [2^e, 2^(e+1)) for normal amax
  const int s = 14 - e;
  return s < -126 ? -126 : (s > 126 ? 126 : s);
}

// Split-K plans: how many K-splits each kernel uses and the workspace it needs.
struct Plan {
  int kernel;            // 0 = GEMV (decode), 1 = FP32 SIMT GEMM, 2 = tcgen05 GEMM (TF32X3 / FP16X3)
  int splits;            // K-splits (1 = none)
  int64_t k_per_split;   // multiple of the kernel's K granule
  size_t ws_partials;    // bytes of split partials (at offset kCounterBytes)
  size_t ws_asplit;      // bytes of the FP16X3 split of A: row exponents, hi, lo (at offset kCounterBytes)
  size_t total() const { return (ws_partials + ws_asplit) ? kCounterBytes + ws_partials + ws_asplit : 0; }
};

constexpr int kGemvMaxM = 16;
constexpr int kKernelGemv = 0, kKernelSimt = 1, kKernelTc = 2;

Plan plan_gemv(int64_t M, int64_t K, int64_t N, int sms);
Plan plan_simt(int64_t M, int64_t K, int64_t N, int sms);
Plan plan_tc(int64_t M, int64_t K, int64_t N, int sms, spl_path path);

spl_status run_gemv(const LinearArgs& a, const Plan& p);
// The decode product with the mask fused into its staging of X~ (a2 + a3 + a5 + a6 in one launch):
// a.a is the unmasked X; X~ = fl32(X + eta) is drawn exactly as spl_noise_mask draws it, used for
// the product and written to nz.xt.  Same plan, same order, same result as the separate calls.
struct MaskNoise {
  float* xt;                   // [M, K] X~ out
  float b;                     // scale Delta f / eps (0: eps = inf, no noise)
  int mech;                    // spl_mech
  uint64_t seed, stream_id;    // Philox key, counter words 2-3
  uint64_t offset;             // Philox block offset (host part)
  const uint64_t* offset_dev;  // device part of the offset (may be null)
  int64_t x_rows = -1;         // rows from x_rows on are noise alone (no X), drawn noise_delta blocks
  uint64_t noise_delta = 0;    // further on with their counters starting again at row x_rows (-1: all rows X)
};
constexpr int kGemvMaskMaxM = 4;  // rows up to which every block draws its slice's noise itself
spl_status run_gemv_masked(const LinearArgs& a, const Plan& p, const MaskNoise& nz);
// Argument check shared by the noise entries.
spl_status validate_noise(int64_t rows, int64_t cols, double sensitivity, double eps, spl_mech mech);
int64_t gemv_max_ks(int64_t M);                           // largest K-slice the decode kernel stages for M rows
// Launch variant and K-split of a one-launch tcgen05 call (false if the call makes two launches);
// variant -1 is the swapped kernel of few rows.
bool tc_uniform_shape(int64_t M, int64_t K, int64_t N, spl_path path, int* variant, int* splits);
// A tcgen05 product whose every output is summed in the order the masked product of `order_rows`
// rows uses (the correction bank): the same K ranges, accumulation chains and cluster order.
spl_status run_tc_matched(const LinearArgs& a, int64_t order_rows);
size_t tc_asplit_bytes(int64_t M, int64_t K, spl_path path);  // FP16X3 split of A in the workspace (0 for TF32X3)
// Workspace for the partial tiles of a tcgen05 product of M rows summed in the order of `order_rows`
// (the swapped kernel's runs; 0 for the cluster-reduced kernels), after the split of A.
size_t tc_partial_bytes(int64_t M, int64_t K, int64_t N, int64_t order_rows, spl_path path);
spl_status run_simt(const LinearArgs& a, const Plan& p);
spl_status run_tc(const LinearArgs& a, const Plan& p);

// Deterministic split-K reduction: out = sum_s part[s] (in s order) - c.
spl_status run_splitk_reduce(float* out, const float* part, const float* c, int splits, int64_t M,
                             int64_t N, cudaStream_t stream);

// Elementwise TF32 split (spl_split_tf32).
spl_status run_split_tf32(float* hi, float* lo, const float* src, int64_t count, cudaStream_t stream);
// Row-scaled fp16 split of a [rows, cols] matrix (spl_split_fp16; the left operand of FP16X3).
spl_status run_split_fp16(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* src, int64_t rows, int64_t cols,
                          cudaStream_t stream);

__host__ __device__ inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
__host__ __device__ inline int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

}  // namespace spl
