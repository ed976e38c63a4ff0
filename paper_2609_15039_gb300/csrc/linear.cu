// Entry points of the product calls: argument checks, path and kernel choice,
// workspace sizing.
//
//   spl_masked_linear             r = X~ W^T            (Sec. 5.1)
//   spl_precompute_noise_product  C = N W^T             (Sec. 5.2)
//   spl_masked_linear_unmask      Y = X~ W^T - C        (Eq. add-and-then-subtract, fused)
//
// Kernel choice: on the FP32 path M <= 16 rows stream W once through the decode
// kernel and larger M use the SIMT kernel.  AUTO takes a tcgen05 kernel for M > 8
// on an sm_100/sm_103 device with K >= 64 (below that the three-product error of
// about 2^-20 per term is not small against gamma_K): FP16X3 when the weight
// descriptor carries the fp16 split and K % 8 == 0, else TF32X3 when it carries the
// TF32 split, else FP32.

#include <algorithm>

#include "common.cuh"

namespace spl {
namespace {

bool tc_capable() {
  const int cc = device_cc();
  return cc == 100 || cc == 103;
}

// AUTO: up to 8 rows the streaming decode kernel reads W once at HBM rate and wins; from
// 9 rows on a tensor-core path is faster even with its 128-row tile mostly empty (the
// decode kernel turns shared-memory bound as M grows).  FP16X3 (4 bytes per weight, twice
// the TF32 rate) is preferred over TF32X3 when its split is present and K % 8 == 0.
constexpr int64_t kAutoDecodeMaxM = 8;

bool has_tf32(const spl_weight& w) { return w.tf32_hi && w.tf32_lo; }
bool has_f16(const spl_weight& w) { return w.f16_hi && w.f16_lo && w.f16_exp; }

spl_path resolve(int64_t M, int64_t K, spl_path path, bool tf32, bool f16) {
  if (path != SPL_PATH_AUTO) return path;
  if (M > kAutoDecodeMaxM && K >= 64 && tc_capable()) {
    if (f16 && (K & 7) == 0) return SPL_PATH_FP16X3;
    if (tf32) return SPL_PATH_TF32X3;
  }
  return SPL_PATH_FP32;
}

bool is_tc(spl_path p) { return p == SPL_PATH_TF32X3 || p == SPL_PATH_FP16X3; }

Plan make_plan(int64_t M, int64_t K, int64_t N, spl_path resolved) {
  const int sms = device_sm_count();
  if (is_tc(resolved)) return plan_tc(M, K, N, sms, resolved);
  if (M <= kGemvMaxM) return plan_gemv(M, K, N, sms);
  return plan_simt(M, K, N, sms);
}

bool valid_path(spl_path p) {
  return p == SPL_PATH_AUTO || p == SPL_PATH_TF32X3 || p == SPL_PATH_FP32 || p == SPL_PATH_FP16X3;
}

spl_status check_weight(const spl_weight* W, int64_t K) {
  if (!W) return SPL_EINVAL;
  if (K > 0 && !W->w) return SPL_EINVAL;
  if (W->w && !aligned16(W->w)) return SPL_EALIGN;
  if ((W->tf32_hi && !aligned16(W->tf32_hi)) || (W->tf32_lo && !aligned16(W->tf32_lo))) return SPL_EALIGN;
  if ((W->f16_hi && !aligned16(W->f16_hi)) || (W->f16_lo && !aligned16(W->f16_lo))) return SPL_EALIGN;
  return SPL_OK;
}

spl_status run_linear(float* out, const float* a, const spl_weight* W, const float* C, bool need_c, int64_t M,
                      int64_t K, int64_t N, spl_path path, void* ws, size_t ws_bytes, cudaStream_t stream,
                      const spl_weight* A = nullptr, const MaskNoise* noise = nullptr, int64_t c_rows = -1) {
  if (M < 0 || K < 0 || N < 0) return SPL_EINVAL;
  if (!valid_path(path)) return SPL_EINVAL;
  if (M == 0 || N == 0) return SPL_OK;
  if (!out || (need_c && !C)) return SPL_EINVAL;
  if ((K & 3) != 0) return SPL_EALIGN;
  spl_status st = check_weight(W, K);
  if (st != SPL_OK) return st;
  // a pre-split left operand (FP16X3): its fp32 values may be absent when that path runs
  const bool a_split = A && A->f16_hi && A->f16_lo && A->f16_exp;
  if (K > 0 && !a && !a_split) return SPL_EINVAL;
  if (!aligned16(out) || (a && !aligned16(a)) || (C && !aligned16(C))) return SPL_EALIGN;
  if (M > (int64_t(1) << 31) || N > (int64_t(1) << 31) || K > (int64_t(1) << 31)) return SPL_ESHAPE;
  if (K == 0) {  // empty reduction: the product is zero
    if (cudaMemsetAsync(out, 0, (size_t)(M * N) * sizeof(float), stream) != cudaSuccess) return SPL_ECUDA;
    return C ? spl_unmask(out, out, C, M, N, stream) : SPL_OK;
  }
  const spl_path resolved = resolve(M, K, path, has_tf32(*W), has_f16(*W));
  if (resolved == SPL_PATH_TF32X3 && (!has_tf32(*W) || !tc_capable())) return SPL_EUNSUPPORTED;
  if (resolved == SPL_PATH_FP16X3 && (!has_f16(*W) || !tc_capable())) return SPL_EUNSUPPORTED;
  if (resolved == SPL_PATH_FP16X3 && (K & 7) != 0) return SPL_EALIGN;
  if (!a && resolved != SPL_PATH_FP16X3) return SPL_EINVAL;  // only FP16X3 reads the split alone
  const bool use_split = a_split && resolved == SPL_PATH_FP16X3;
  const Plan plan = make_plan(M, K, N, resolved);
  // a pre-split operand needs only the counters and partial tiles (the split of A is not written)
  const size_t need = use_split ? (plan.ws_partials ? kCounterBytes + plan.ws_partials : 0) : plan.total();
  if (need > 0 && (!ws || ws_bytes < need)) return SPL_EWORKSPACE;
  if (ws && !aligned16(ws)) return SPL_EALIGN;
  LinearArgs args = make_args(out, a, *W, C, M, K, N, ws, ws_bytes, stream, resolved);
  if (c_rows >= 0) {  // only the first c_rows output rows subtract C (tensor-core and decode kernels)
    if (plan.kernel != kKernelTc && plan.kernel != kKernelGemv) return SPL_EUNSUPPORTED;
    args.c_rows = c_rows;
  }
  if (use_split) {
    args.a_h16 = A->f16_hi;
    args.a_l16 = A->f16_lo;
    args.a_exp = A->f16_exp;
  }
  if (noise && (plan.kernel != kKernelGemv || M > kGemvMaskMaxM)) return SPL_EUNSUPPORTED;
  switch (plan.kernel) {
    case kKernelTc: return run_tc(args, plan);
    case kKernelGemv: return noise ? run_gemv_masked(args, plan, *noise) : run_gemv(args, plan);
    default: return run_simt(args, plan);
  }
}

// The plan a correction of M rows must follow so that every output element is summed in the
// order a masked product of `order_rows` rows uses (same kernel, same K-split boundaries, same
// order of the cross-CTA reduction).  ok = false when that order cannot be reproduced.
struct MatchedPlan {
  bool ok;
  int kernel;
  int splits;
  int64_t k_per_split;
  int64_t chunk_rows;  // decode kernel: rows per launch (<= 16)
  size_t ws;           // workspace bytes
};

MatchedPlan matched_plan(int64_t M, int64_t K, int64_t N, int64_t order_rows, spl_path resolved) {
  MatchedPlan mp{false, 0, 1, K, M, 0};
  const Plan online = make_plan(order_rows, K, N, resolved);
  mp.kernel = online.kernel;
  if (online.kernel == kKernelTc) {
    int variant = 0;  // the bank runs its own launch shape; only the K-split order carries over
    if (!tc_uniform_shape(order_rows, K, N, resolved, &variant, &mp.splits)) return mp;
    mp.ws = kCounterBytes + tc_asplit_bytes(M, K, resolved) + tc_partial_bytes(M, K, N, order_rows, resolved);
    mp.ok = true;
    return mp;
  }
  mp.splits = online.splits;
  mp.k_per_split = online.k_per_split;
  if (online.kernel == kKernelGemv) {
    // rows per launch: the most (a power of two up to 16) whose shared-memory K-slice still holds
    // the online K-split; a row's sum does not depend on how many rows a launch carries
    mp.chunk_rows = 0;
    for (int64_t c = kGemvMaxM; c >= 1 && mp.chunk_rows == 0; c /= 2)
      if (c <= std::max<int64_t>(M, 1) && gemv_max_ks(c) >= mp.k_per_split) mp.chunk_rows = std::min<int64_t>(c, M);
    if (mp.chunk_rows == 0) return mp;
    if (mp.splits > 1) mp.ws = kCounterBytes + (size_t)round_up((int64_t)mp.splits * mp.chunk_rows * N * 4, 256);
  } else {
    if (mp.splits > 1) mp.ws = kCounterBytes + (size_t)round_up((int64_t)mp.splits * M * N * 4, 256);
  }
  mp.ok = true;
  return mp;
}

// Workspace of a product call for every path it could take (AUTO: all of them).
size_t linear_ws(int64_t M, int64_t K, int64_t N, spl_path path) {
  size_t need = 0;
  const spl_path paths[3] = {SPL_PATH_FP32, SPL_PATH_TF32X3, SPL_PATH_FP16X3};
  for (spl_path p : paths)
    if (path == SPL_PATH_AUTO || path == p) need = std::max(need, make_plan(M, K, N, p).total());
  return need;
}

}  // namespace
}  // namespace spl

using namespace spl;

extern "C" spl_path spl_resolve_path(int64_t M, int64_t K, int64_t N, spl_path path) {
  (void)N;
  return resolve(M, K, path, true, true);
}

extern "C" size_t spl_linear_workspace_bytes(int64_t M, int64_t K, int64_t N, spl_path path) {
  if (M <= 0 || K <= 0 || N <= 0) return 0;
  return linear_ws(M, K, N, path);
}

extern "C" spl_status spl_masked_linear(float* Yt, const float* Xt, const spl_weight* W, int64_t M, int64_t K,
                                        int64_t N, spl_path path, void* workspace, size_t workspace_bytes,
                                        cudaStream_t stream) {
  return run_linear(Yt, Xt, W, nullptr, false, M, K, N, path, workspace, workspace_bytes, stream);
}

extern "C" spl_status spl_precompute_noise_product(float* C, const float* Nz, const spl_weight* W, int64_t M,
                                                   int64_t K, int64_t N, spl_path path, void* workspace,
                                                   size_t workspace_bytes, cudaStream_t stream) {
  return run_linear(C, Nz, W, nullptr, false, M, K, N, path, workspace, workspace_bytes, stream);
}

extern "C" spl_status spl_masked_linear_unmask(float* Y, const float* Xt, const spl_weight* W, const float* C,
                                               int64_t M, int64_t K, int64_t N, spl_path path, void* workspace,
                                               size_t workspace_bytes, cudaStream_t stream) {
  return run_linear(Y, Xt, W, C, true, M, K, N, path, workspace, workspace_bytes, stream);
}

extern "C" spl_status spl_masked_linear_unmask_split(float* Y, const spl_weight* Xt, const spl_weight* W,
                                                     const float* C, int64_t M, int64_t K, int64_t N, spl_path path,
                                                     void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  if (!Xt) return SPL_EINVAL;
  return run_linear(Y, Xt->w, W, C, true, M, K, N, path, workspace, workspace_bytes, stream, Xt);
}

extern "C" spl_status spl_masked_linear_unmask_precompute(float* YC, const spl_weight* A, const spl_weight* W,
                                                          const float* C, int64_t M, int64_t M_bank, int64_t K,
                                                          int64_t N, spl_path path, void* workspace,
                                                          size_t workspace_bytes, cudaStream_t stream) {
  if (!A || M < 0 || M_bank < 0) return SPL_EINVAL;
  if (M > 0 && !C) return SPL_EINVAL;
  if (M + M_bank > (int64_t(1) << 31)) return SPL_ESHAPE;
  if (M + M_bank == 0 || N == 0) return SPL_OK;
  if (K > 0) {  // the tensor-core kernels and the decode kernel: decide before anything runs
    const spl_path resolved = resolve(M + M_bank, K, path, W && has_tf32(*W), W && has_f16(*W));
    if (!is_tc(resolved) && M + M_bank > kGemvMaxM) return SPL_EUNSUPPORTED;
  }
  return run_linear(YC, A->w, W, C, M > 0, M + M_bank, K, N, path, workspace, workspace_bytes, stream, A, nullptr,
                    M);
}

extern "C" spl_status spl_noise_mask_linear_unmask_precompute(float* YC, float* Xt, const float* X,
                                                               const spl_weight* W, const float* C, int64_t M,
                                                               int64_t M_bank, int64_t K, int64_t N,
                                                               double sensitivity, double eps, spl_mech mech,
                                                               spl_rng rng, uint64_t noise_block_delta,
                                                               spl_path path, void* workspace, size_t workspace_bytes,
                                                               cudaStream_t stream) {
  spl_status st = validate_noise(M, K, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  if (M_bank < 0 || N < 0 || !valid_path(path)) return SPL_EINVAL;
  const int64_t rows = M + M_bank;
  if (rows == 0 || N == 0) return SPL_OK;
  if (K > 0 && (!Xt || (M > 0 && !X) || !W)) return SPL_EINVAL;
  if (M > 0 && !C) return SPL_EINVAL;
  if ((Xt && !aligned16(Xt)) || (X && !aligned16(X))) return SPL_EALIGN;
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  if (K == 0 || rows > kGemvMaskMaxM || resolve(rows, K, path, has_tf32(*W), has_f16(*W)) != SPL_PATH_FP32)
    return SPL_EUNSUPPORTED;  // one launch on the decode kernel only
  if (X && M > 0) {  // X~ is written while other blocks still read X
    const uintptr_t x0 = reinterpret_cast<uintptr_t>(X), t0 = reinterpret_cast<uintptr_t>(Xt);
    const uintptr_t xb = (uintptr_t)(M * K) * sizeof(float), tb = (uintptr_t)(rows * K) * sizeof(float);
    if (x0 < t0 + tb && t0 < x0 + xb) return SPL_EINVAL;
  }
  MaskNoise nz{};
  nz.xt = Xt;
  nz.b = std::isinf(eps) ? 0.0f : (float)(sensitivity / eps);
  nz.mech = (int)mech;
  nz.seed = rng.seed;
  nz.stream_id = rng.stream_id;
  nz.offset = rng.offset;
  nz.offset_dev = rng.offset_dev;
  nz.x_rows = M;
  nz.noise_delta = noise_block_delta;
  return run_linear(YC, X ? X : Xt, W, C, M > 0, rows, K, N, path, workspace, workspace_bytes, stream, nullptr, &nz,
                    M);
}

extern "C" spl_status spl_noise_mask_linear_unmask(float* Y, float* Xt, const float* X, const spl_weight* W,
                                                   const float* C, int64_t M, int64_t K, int64_t N,
                                                   double sensitivity, double eps, spl_mech mech, spl_rng rng,
                                                   spl_path path, void* workspace, size_t workspace_bytes,
                                                   cudaStream_t stream) {
  spl_status st = validate_noise(M, K, sensitivity, eps, mech);
  if (st != SPL_OK) return st;
  if (N < 0 || !valid_path(path)) return SPL_EINVAL;
  if (M > 0 && K > 0 && (!Xt || !X)) return SPL_EINVAL;
  if ((Xt && !aligned16(Xt)) || (X && !aligned16(X))) return SPL_EALIGN;
  if ((reinterpret_cast<uintptr_t>(rng.offset_dev) & 7u) != 0) return SPL_EALIGN;
  if (M > 0 && K > 0) {  // X~ is written while other blocks still read X
    const uintptr_t x0 = reinterpret_cast<uintptr_t>(X), t0 = reinterpret_cast<uintptr_t>(Xt);
    const uintptr_t bytes = (uintptr_t)(M * K) * sizeof(float);
    if (x0 < t0 + bytes && t0 < x0 + bytes) return SPL_EINVAL;
  }
  const bool fused = M > 0 && M <= kGemvMaskMaxM && K > 0 && N > 0 && W &&
                     resolve(M, K, path, has_tf32(*W), has_f16(*W)) == SPL_PATH_FP32;
  if (!fused) {  // mask, then the product: two launches with the same results
    st = spl_noise_mask(Xt, nullptr, X, M, K, sensitivity, eps, mech, rng, stream);
    if (st != SPL_OK) return st;
    return run_linear(Y, Xt, W, C, true, M, K, N, path, workspace, workspace_bytes, stream);
  }
  MaskNoise nz{};
  nz.xt = Xt;
  nz.b = std::isinf(eps) ? 0.0f : (float)(sensitivity / eps);
  nz.mech = (int)mech;
  nz.seed = rng.seed;
  nz.stream_id = rng.stream_id;
  nz.offset = rng.offset;
  nz.offset_dev = rng.offset_dev;
  return run_linear(Y, X, W, C, true, M, K, N, path, workspace, workspace_bytes, stream, nullptr, &nz);
}

extern "C" size_t spl_split_workspace_bytes(int64_t M, int64_t K, int64_t N, int64_t order_rows, spl_path path) {
  if (M <= 0 || K <= 0 || N <= 0 || order_rows <= 0 || !valid_path(path)) return 0;
  size_t need = 0;
  const spl_path paths[3] = {SPL_PATH_FP32, SPL_PATH_TF32X3, SPL_PATH_FP16X3};
  for (spl_path p : paths) {
    if (path != SPL_PATH_AUTO && path != p) continue;
    if (p == SPL_PATH_FP16X3) {  // the split is read as given: counters and partial tiles only
      const size_t part = tc_partial_bytes(M, K, N, order_rows, p);
      need = std::max(need, part ? kCounterBytes + part : (size_t)0);
    } else {  // these paths read the fp32 operand
      const MatchedPlan mp = matched_plan(M, K, N, order_rows, p);
      need = std::max(need, order_rows == M ? make_plan(M, K, N, p).total() : (mp.ok ? mp.ws : make_plan(M, K, N, p).total()));
    }
  }
  return need;
}

extern "C" size_t spl_precompute_matched_workspace_bytes(int64_t M, int64_t K, int64_t N, int64_t order_rows,
                                                         spl_path path) {
  if (M <= 0 || K <= 0 || N <= 0 || order_rows <= 0) return 0;
  size_t need = 0;
  const spl_path paths[3] = {SPL_PATH_FP32, SPL_PATH_TF32X3, SPL_PATH_FP16X3};
  for (spl_path p : paths) {
    if (path != SPL_PATH_AUTO && path != p) continue;
    const MatchedPlan mp = matched_plan(M, K, N, order_rows, p);
    need = std::max(need, mp.ok ? mp.ws : make_plan(M, K, N, p).total());
  }
  return need;
}

namespace spl {
namespace {
// The correction in the online order; A (may be NULL) carries the fp16 split of the noise.
spl_status precompute_matched(float* C, const float* Nz, const spl_weight* A, const spl_weight* W, int64_t M,
                              int64_t K, int64_t N, int64_t order_rows, spl_path path, void* workspace,
                              size_t workspace_bytes, cudaStream_t stream) {
  if (order_rows <= 0) return SPL_EINVAL;
  if (M < 0 || K < 0 || N < 0) return SPL_EINVAL;
  if (!valid_path(path)) return SPL_EINVAL;
  if (M == 0 || N == 0 || K == 0)
    return run_linear(C, Nz, W, nullptr, false, M, K, N, path, workspace, workspace_bytes, stream, A);
  const bool a_split = A && A->f16_hi && A->f16_lo && A->f16_exp;
  if (!C || (!Nz && !a_split)) return SPL_EINVAL;
  spl_status st = check_weight(W, K);
  if (st != SPL_OK) return st;
  if ((K & 3) != 0) return SPL_EALIGN;
  if (!aligned16(C) || (Nz && !aligned16(Nz))) return SPL_EALIGN;
  const spl_path resolved = resolve(order_rows, K, path, has_tf32(*W), has_f16(*W));
  if (resolved == SPL_PATH_TF32X3 && (!has_tf32(*W) || !tc_capable())) return SPL_EUNSUPPORTED;
  if (resolved == SPL_PATH_FP16X3 && (!has_f16(*W) || !tc_capable())) return SPL_EUNSUPPORTED;
  if (resolved == SPL_PATH_FP16X3 && (K & 7) != 0) return SPL_EALIGN;
  const bool use_split = a_split && resolved == SPL_PATH_FP16X3;
  if (!Nz && !use_split) return SPL_EINVAL;  // only FP16X3 reads the split alone
  const MatchedPlan mp = matched_plan(M, K, N, order_rows, resolved);
  if (!mp.ok)  // the masked call's order cannot be reproduced: plain correction
    return run_linear(C, Nz, W, nullptr, false, M, K, N, resolved, workspace, workspace_bytes, stream, A);
  if (mp.ws > 0 && (!workspace || workspace_bytes < mp.ws)) return SPL_EWORKSPACE;
  if (workspace && !aligned16(workspace)) return SPL_EALIGN;
  LinearArgs args = make_args(C, Nz, *W, nullptr, M, K, N, workspace, workspace_bytes, stream, resolved);
  if (use_split) {
    args.a_h16 = A->f16_hi;
    args.a_l16 = A->f16_lo;
    args.a_exp = A->f16_exp;
  }
  if (mp.kernel == kKernelTc) return run_tc_matched(args, order_rows);
  Plan p{};
  p.kernel = mp.kernel;
  p.splits = mp.splits;
  p.k_per_split = mp.k_per_split;
  if (mp.kernel == kKernelSimt) {
    p.ws_partials = mp.splits > 1 ? (size_t)round_up((int64_t)mp.splits * M * N * 4, 256) : 0;
    return run_simt(args, p);
  }
  for (int64_t r0 = 0; r0 < M; r0 += mp.chunk_rows) {  // decode kernel: at most 16 rows per launch
    const int64_t rows = std::min<int64_t>(mp.chunk_rows, M - r0);
    const LinearArgs ca = make_args(C + r0 * N, Nz + r0 * K, *W, nullptr, rows, K, N, workspace, workspace_bytes,
                                    stream, resolved);
    p.ws_partials = mp.splits > 1 ? (size_t)round_up((int64_t)mp.splits * rows * N * 4, 256) : 0;
    st = run_gemv(ca, p);
    if (st != SPL_OK) return st;
  }
  return SPL_OK;
}
}  // namespace
}  // namespace spl

extern "C" spl_status spl_precompute_noise_product_matched(float* C, const float* Nz, const spl_weight* W, int64_t M,
                                                           int64_t K, int64_t N, int64_t order_rows, spl_path path,
                                                           void* workspace, size_t workspace_bytes,
                                                           cudaStream_t stream) {
  if (M > 0 && K > 0 && N > 0 && !Nz) return SPL_EINVAL;
  return precompute_matched(C, Nz, nullptr, W, M, K, N, order_rows, path, workspace, workspace_bytes, stream);
}

extern "C" spl_status spl_precompute_noise_product_matched_split(float* C, const spl_weight* Nz, const spl_weight* W,
                                                                 int64_t M, int64_t K, int64_t N, int64_t order_rows,
                                                                 spl_path path, void* workspace,
                                                                 size_t workspace_bytes, cudaStream_t stream) {
  if (!Nz) return SPL_EINVAL;
  return precompute_matched(C, Nz->w, Nz, W, M, K, N, order_rows, path, workspace, workspace_bytes, stream);
}
