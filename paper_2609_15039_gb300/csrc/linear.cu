// Entry points of the product calls: argument checks, path and kernel choice,
// workspace sizing.
//
//   spl_masked_linear             r = X~ W^T            (Sec. 5.1)
//   spl_precompute_noise_product  C = N W^T             (Sec. 5.2)
//   spl_masked_linear_unmask      Y = X~ W^T - C        (Eq. add-and-then-subtract, fused)
//
// Kernel choice: on the FP32 path M <= 16 rows stream W once through the decode
// kernel and larger M use the SIMT kernel.  AUTO takes the TF32X3 tcgen05
// kernel for M > 8 when the weight split is available, the device is
// sm_100/sm_103 and K >= 64 (below that the three-product error of about
// 2^-20 per term is not small against gamma_K), else FP32.

#include <algorithm>

#include "common.cuh"

namespace spl {
namespace {

bool tc_capable() {
  const int cc = device_cc();
  return cc == 100 || cc == 103;
}

// AUTO: up to 8 rows the streaming decode kernel reads W once at HBM rate and
// wins; from 9 rows on the tensor-core kernel is faster even with its 128-row
// tile mostly empty (the decode kernel turns shared-memory bound as M grows).
constexpr int64_t kAutoDecodeMaxM = 8;

spl_path resolve(int64_t M, int64_t K, spl_path path, bool have_split) {
  if (path == SPL_PATH_FP32 || path == SPL_PATH_TF32X3) return path;
  if (M > kAutoDecodeMaxM && K >= 64 && have_split && tc_capable()) return SPL_PATH_TF32X3;
  return SPL_PATH_FP32;
}

Plan make_plan(int64_t M, int64_t K, int64_t N, spl_path resolved) {
  const int sms = device_sm_count();
  if (resolved == SPL_PATH_TF32X3) return plan_tc(M, K, N, sms);
  if (M <= kGemvMaxM) return plan_gemv(M, K, N, sms);
  return plan_simt(M, K, N, sms);
}

spl_status run_linear(float* out, const float* a, const float* W, const float* W_hi, const float* W_lo,
                      const float* C, bool need_c, int64_t M, int64_t K, int64_t N, spl_path path, void* ws,
                      size_t ws_bytes, cudaStream_t stream) {
  if (M < 0 || K < 0 || N < 0) return SPL_EINVAL;
  if (path != SPL_PATH_AUTO && path != SPL_PATH_TF32X3 && path != SPL_PATH_FP32) return SPL_EINVAL;
  if (M == 0 || N == 0) return SPL_OK;
  if (!out || (need_c && !C)) return SPL_EINVAL;
  if ((K & 3) != 0) return SPL_EALIGN;
  if (K > 0 && (!a || !W)) return SPL_EINVAL;
  if (!aligned16(out) || (a && !aligned16(a)) || (W && !aligned16(W)) || (C && !aligned16(C))) return SPL_EALIGN;
  if ((W_hi && !aligned16(W_hi)) || (W_lo && !aligned16(W_lo))) return SPL_EALIGN;
  if (M > (int64_t(1) << 31) || N > (int64_t(1) << 31) || K > (int64_t(1) << 31)) return SPL_ESHAPE;
  if (K == 0) {  // empty reduction: the product is zero
    if (cudaMemsetAsync(out, 0, (size_t)(M * N) * sizeof(float), stream) != cudaSuccess) return SPL_ECUDA;
    return C ? spl_unmask(out, out, C, M, N, stream) : SPL_OK;
  }
  const spl_path resolved = resolve(M, K, path, W_hi && W_lo);
  if (resolved == SPL_PATH_TF32X3 && (!W_hi || !W_lo || !tc_capable())) return SPL_EUNSUPPORTED;
  const Plan plan = make_plan(M, K, N, resolved);
  if (plan.total() > 0 && (!ws || ws_bytes < plan.total())) return SPL_EWORKSPACE;
  if (ws && !aligned16(ws)) return SPL_EALIGN;
  LinearArgs args{out, a, W, W_hi, W_lo, C, M, K, N, ws, ws_bytes, stream};
  switch (plan.kernel) {
    case kKernelTc: return run_tc(args, plan);
    case kKernelGemv: return run_gemv(args, plan);
    default: return run_simt(args, plan);
  }
}

}  // namespace
}  // namespace spl

using namespace spl;

extern "C" spl_path spl_resolve_path(int64_t M, int64_t K, int64_t N, spl_path path) {
  (void)N;
  return resolve(M, K, path, true);
}

extern "C" size_t spl_linear_workspace_bytes(int64_t M, int64_t K, int64_t N, spl_path path) {
  if (M <= 0 || K <= 0 || N <= 0) return 0;
  size_t need = 0;
  if (path == SPL_PATH_AUTO || path == SPL_PATH_FP32) need = std::max(need, make_plan(M, K, N, SPL_PATH_FP32).total());
  if (path == SPL_PATH_AUTO || path == SPL_PATH_TF32X3)
    need = std::max(need, make_plan(M, K, N, SPL_PATH_TF32X3).total());
  return need;
}

extern "C" spl_status spl_masked_linear(float* Yt, const float* Xt, const float* W, const float* W_hi,
                                        const float* W_lo, int64_t M, int64_t K, int64_t N, spl_path path,
                                        void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  return run_linear(Yt, Xt, W, W_hi, W_lo, nullptr, false, M, K, N, path, workspace, workspace_bytes, stream);
}

extern "C" spl_status spl_precompute_noise_product(float* C, const float* Nz, const float* W, const float* W_hi,
                                                   const float* W_lo, int64_t M, int64_t K, int64_t N,
                                                   spl_path path, void* workspace, size_t workspace_bytes,
                                                   cudaStream_t stream) {
  return run_linear(C, Nz, W, W_hi, W_lo, nullptr, false, M, K, N, path, workspace, workspace_bytes, stream);
}

extern "C" spl_status spl_masked_linear_unmask(float* Y, const float* Xt, const float* W, const float* W_hi,
                                               const float* W_lo, const float* C, int64_t M, int64_t K, int64_t N,
                                               spl_path path, void* workspace, size_t workspace_bytes,
                                               cudaStream_t stream) {
  return run_linear(Y, Xt, W, W_hi, W_lo, C, true, M, K, N, path, workspace, workspace_bytes, stream);
}
