/*
 * spl.h -- C ABI of the SpliTEE masked-linear hot path on GB300 (sm_103a).
 *
 * The method (arxiv 2609.15039, Sec. 3.3.1 and Eq. add-and-then-subtract):
 * a trusted party masks the input x of a linear layer with differentially
 * private noise eta, x~ = x + eta; the untrusted GPU computes r = W x~; the
 * result is unmasked with the precomputed correction W eta,
 * W x = r - W eta.  The noise follows the Gaussian mechanism with scale
 * Delta f / eps (Prop. eps-GDP mechanism, Sec. 4.4); a Laplace variant with
 * the same scale is also offered.  Delta f comes from Thms. 1-3 (Sec. 4.3).
 *
 * Conventions for every call
 *  - Tensors are fp32, row-major and contiguous.  Rows are tokens.
 *    X, X~ and the noise N are [M, K]; weights W are [N, K] (K contiguous,
 *    the nn.Linear layout); outputs are [M, N].  The paper writes the same
 *    product with column vectors (W x); here it is X W^T.
 *  - Device pointers are owned by the caller.  Every base pointer must be
 *    16-byte aligned and K must be a multiple of 4 (SPL_EALIGN otherwise).
 *  - Work is enqueued asynchronously on `stream` (0 = legacy default stream);
 *    no call synchronises the host except spl_get_device_status and
 *    spl_spectral_norm.  A zero-sized problem returns SPL_OK and does nothing.
 *  - Arguments are validated before anything is launched; an invalid call
 *    launches nothing.  Launch failures return SPL_ECUDA.
 *  - The library keeps no allocation of its own beyond one device status
 *    word (set by kernels whose bounded waits expire, read by
 *    spl_get_device_status).  Scratch memory is passed in as `workspace`.
 */
#ifndef SPL_H
#define SPL_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum spl_status {
  SPL_OK = 0,
  SPL_EINVAL = 1,       /* invalid value: NULL pointer, eps <= 0 or NaN, negative size, bad enum */
  SPL_ESHAPE = 2,       /* sizes out of the supported range */
  SPL_EALIGN = 3,       /* base pointer not 16-byte aligned, or K % 4 != 0 */
  SPL_ECUDA = 4,        /* a CUDA runtime or driver call failed */
  SPL_ETIMEOUT = 5,     /* a bounded device-side wait expired (see spl_get_device_status) */
  SPL_EUNSUPPORTED = 6, /* the requested path cannot run on this device or with these operands */
  SPL_EWORKSPACE = 7    /* workspace missing or smaller than spl_linear_workspace_bytes() */
} spl_status;

/* Noise law.  GAUSSIAN is the paper's mechanism (Sec. 4.4); LAPLACE uses the
 * same scale b = Delta f / eps. */
typedef enum spl_mech { SPL_MECH_LAPLACE = 0, SPL_MECH_GAUSSIAN = 1 } spl_mech;

/* Arithmetic of the masked product.
 *  FP32   -- fp32 FMA on the CUDA cores (each product exact before its
 *            rounding, sequential summation per output).
 *  TF32X3 -- tcgen05 tensor cores, three TF32 products per term
 *            (hi*hi + hi*lo + lo*hi, fp32 accumulation in TMEM); needs the
 *            weight split of spl_split_tf32 (8 bytes per weight).
 *  FP16X3 -- the same three products in fp16 (kind::f16, twice the TF32 rate)
 *            on rows scaled by powers of two, undone exactly in the epilogue;
 *            needs the weight split of spl_split_fp16 (4 bytes per weight)
 *            and K % 8 == 0.  Per-term error about 2^-21 |a w| plus an
 *            absolute 2^-39 max|a_row| |w| for entries that fall below fp16's
 *            normal range after the row scaling (more than ~2^-28 under the
 *            row's largest); spl_choose_path judges whether that stays inside
 *            the bound for the data at hand.
 *  AUTO   -- the library's choice (spl_resolve_path). */
typedef enum spl_path {
  SPL_PATH_AUTO = 0,
  SPL_PATH_TF32X3 = 1,
  SPL_PATH_FP32 = 2,
  SPL_PATH_FP16X3 = 3
} spl_path;

/* A weight W[N, K] (fp32, K contiguous) and the splits the tensor-core paths
 * read.  Device pointers owned by the caller; any split may be NULL (the
 * paths that need it then report SPL_EUNSUPPORTED and AUTO skips them). */
typedef struct spl_weight {
  const float* w;          /* [N, K] fp32, required */
  const float* tf32_hi;    /* [N, K] from spl_split_tf32 */
  const float* tf32_lo;
  const uint16_t* f16_hi;  /* [N, K] binary16 bit patterns from spl_split_fp16 */
  const uint16_t* f16_lo;
  const int32_t* f16_exp;  /* [N] power-of-two row exponents of the fp16 split */
} spl_weight;

/* Philox4x32-10 stream (Salmon et al., SC'11).  Element e of a flat tensor
 * uses lane e % 4 of block j = e / 4 + offset (64-bit, wrapping); the
 * counter is (lo32 j, hi32 j, lo32 stream_id, hi32 stream_id) and the key
 * (lo32 seed, hi32 seed).  Distinct (seed, stream_id, block) never share a
 * counter, so draws with disjoint block ranges are independent. */
typedef struct spl_rng {
  uint64_t seed;
  uint64_t stream_id;
  uint64_t offset;
  /* Optional DEVICE pointer (8-byte aligned) or NULL: the kernel adds the value it
   * finds there, when it runs, to `offset`.  A CUDA graph captured with it draws
   * fresh noise on every replay once the value is moved on (spl_rng_advance). */
  const uint64_t* offset_dev;
} spl_rng;

/* ---- a2: noise --------------------------------------------------------
 * N[rows, cols] <- eta, scale b = fl32(sensitivity / eps) (Sec. 4.4).
 *  Laplace: per element one word r; sign = bit 31, u = ((r & 0xFFFFFF)+1) 2^-24,
 *           eta = +-b (-ln u).
 *  Gaussian: Box-Muller on word pairs (0,1), (2,3) of a block:
 *           u1 = ((r_a >> 8)+1) 2^-24, u2 = (r_b >> 8) 2^-24,
 *           eta_a = b R cos(2 pi u2), eta_b = b R sin(2 pi u2), R = sqrt(-2 ln u1).
 * eps = +INFINITY writes zeros (the noise-free T3 configuration).
 * Errors: EINVAL if N is NULL, eps <= 0 or NaN, sensitivity < 0 or not finite,
 * or mech unknown; EALIGN if N is not 16-byte aligned. */
spl_status spl_noise(float* N, int64_t rows, int64_t cols, double sensitivity, double eps,
                     spl_mech mech, spl_rng rng, cudaStream_t stream);

/* The raw 32-bit words of the Philox stream above: out[e] is lane e % 4 of
 * block e / 4 + rng.offset.  This is the integer stream spl_noise transforms.
 * Errors: EINVAL for NULL out or count < 0, EALIGN if out is not 16-byte aligned. */
spl_status spl_random_bits(uint32_t* out, int64_t count, spl_rng rng, cudaStream_t stream);

/* *offset_dev += delta, on the device, in stream order (one thread).  The step a
 * captured graph ends with to move its draws to the next blocks of the stream.
 * Errors: EINVAL for NULL, EALIGN if not 8-byte aligned. */
spl_status spl_rng_advance(uint64_t* offset_dev, uint64_t delta, cudaStream_t stream);

/* ---- a3: mask ---------------------------------------------------------
 * Xt = fl32(X + N) elementwise, round-to-nearest (Sec. 3.3.1).  Xt may alias X. */
spl_status spl_mask(float* Xt, const float* X, const float* N, int64_t rows, int64_t cols,
                    cudaStream_t stream);

/* ---- a2 + a3 fused ----------------------------------------------------
 * Draws eta exactly as spl_noise and writes Xt = fl32(X + eta) in one pass.
 * N_out (may be NULL) receives eta for the correction precompute.
 * Xt may alias X.  Same errors as spl_noise plus EINVAL for NULL X / Xt. */
spl_status spl_noise_mask(float* Xt, float* N_out, const float* X, int64_t rows, int64_t cols,
                          double sensitivity, double eps, spl_mech mech, spl_rng rng,
                          cudaStream_t stream);

/* ---- a2 + a3 fused with the fp16 split of X~ ----------------------------
 * Draws eta exactly as spl_noise, forms Xt = fl32(X + eta) (written to Xt
 * unless it is NULL) and writes its FP16X3 split as spl_split_fp16 would:
 * hi, lo [rows, cols] binary16 and row_exp [rows].  With X NULL the split is
 * that of eta itself (and Xt, if given, receives eta): a bank of noise draws
 * split in one pass for spl_precompute_noise_product_matched_split.  One pass,
 * one block per row; cols % 8 == 0 and cols <= 16384 (EALIGN / ESHAPE
 * otherwise).  The split is what spl_masked_linear_unmask_split consumes.
 * Errors as spl_noise_mask, except that X may be NULL. */
spl_status spl_noise_mask_split(float* Xt, uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* X,
                                int64_t rows, int64_t cols, double sensitivity, double eps, spl_mech mech,
                                spl_rng rng, cudaStream_t stream);

/* The left operand of spl_masked_linear_unmask_precompute in one pass: rows
 * 0..x_rows-1 of hi / lo / row_exp get the split of fl32(X + eta), eta drawn
 * as spl_noise_mask_split draws it for X (block offset rng.offset, rows from
 * 0); rows x_rows..x_rows+noise_rows-1 get the split of noise alone, drawn as
 * spl_noise_mask_split with X NULL would draw noise_rows rows at block offset
 * rng.offset + noise_block_delta (e.g. the same draw of the next bank cycle).
 * Bit for bit the two separate calls, in one launch.  X [x_rows, cols];
 * hi, lo [x_rows + noise_rows, cols], row_exp [x_rows + noise_rows].  Errors
 * as spl_noise_mask_split (EINVAL for NULL X with x_rows > 0 or negative
 * counts). */
spl_status spl_noise_mask_split_stacked(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* X,
                                        int64_t x_rows, int64_t noise_rows, int64_t cols, double sensitivity,
                                        double eps, spl_mech mech, spl_rng rng, uint64_t noise_block_delta,
                                        cudaStream_t stream);

/* ---- a3 with a stored noise, fused with the fp16 split of X~ -------------
 * Xt = fl32(X + N) elementwise (Sec. 3.3.1, the mask with a noise drawn earlier,
 * e.g. written by spl_noise_mask_split with X NULL while a bank of corrections
 * was precomputed), written to Xt unless it is NULL, and its FP16X3 split as
 * spl_split_fp16 would write it: hi, lo [rows, cols] binary16 and row_exp
 * [rows].  With N = the noise spl_noise_mask_split draws for the same rows, the
 * outputs equal spl_noise_mask_split's bit for bit.  X, N [rows, cols] fp32,
 * device, not aliasing the outputs.  One pass, one block per row.  Errors:
 * EINVAL for negative sizes or NULL hi / lo / row_exp / X / N; EALIGN for
 * cols % 8 != 0 or a pointer not 16-byte aligned; ESHAPE for cols > 16384. */
spl_status spl_mask_split(float* Xt, uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* X,
                          const float* N, int64_t rows, int64_t cols, cudaStream_t stream);

/* ---- weight preparation for TF32X3 ------------------------------------
 * hi = src rounded to TF32 (10 explicit mantissa bits, ties away), lo = src - hi
 * (exact in fp32).  Done once per weight; hi and lo are [count] like src. */
spl_status spl_split_tf32(float* hi, float* lo, const float* src, int64_t count, cudaStream_t stream);

/* hi = fp16(src 2^e_r), lo = fp16(src 2^e_r - hi) per row r, with the power of
 * two e_r (row_exp[r]) that brings the row's largest |entry| into [2^14, 2^15)
 * (0 for an all-zero row); hi + lo = src 2^e_r to about 2^-22 relative.  Done
 * once per weight; hi and lo are [rows, cols] binary16 bit patterns.
 * cols % 8 == 0 (EALIGN otherwise). */
spl_status spl_split_fp16(uint16_t* hi, uint16_t* lo, int32_t* row_exp, const float* src, int64_t rows,
                          int64_t cols, cudaStream_t stream);

/* Path that AUTO resolves to for an M x K x N product on the current device,
 * assuming every split is passed: FP32 up to 8 rows (the streaming decode
 * kernel), else FP16X3 when K % 8 == 0, else TF32X3 (K >= 64, tcgen05 device),
 * else FP32.  An explicit path is returned unchanged. */
spl_path spl_resolve_path(int64_t M, int64_t K, int64_t N, spl_path path);

/* Bytes of device workspace the three product calls below need for this
 * problem on the current device (0 if none; for AUTO the largest over the
 * paths).  Layout: the first 64 KiB hold the arrival counters of the decode
 * kernel and of the swapped few-row kernel, then either split-K partial sums
 * (FP32 kernels) or the split of the left operand for the tensor-core paths
 * (TF32X3: hi and lo in fp32; FP16X3: one power-of-two exponent per row, hi
 * and lo in fp16), followed for 9-16 rows on FP16X3 by the swapped kernel's
 * partial tiles.  It must be zero-filled before its first use; every call that
 * returns SPL_OK leaves the counters at zero again, so one workspace (sized
 * for the largest call) serves calls of any shape and path.  After a call
 * whose kernels gave up a bounded wait (spl_get_device_status returns
 * SPL_ETIMEOUT) the counters may not be zero: zero the first 64 KiB again
 * before the workspace is reused.  Calls that can run concurrently must not
 * share a workspace. */
size_t spl_linear_workspace_bytes(int64_t M, int64_t K, int64_t N, spl_path path);

/* ---- a5: masked product -----------------------------------------------
 * Yt[M, N] = Xt[M, K] W[N, K]^T, the GPU's r = W x~ (Sec. 5.1).  W carries the
 * fp32 weight and whichever splits exist; AUTO uses only the ones present.
 * Errors: EINVAL for NULL operands, EALIGN, EUNSUPPORTED for a tensor-core path
 * whose split is missing or on a device that is not sm_103/sm_100, EALIGN for
 * FP16X3 with K % 8 != 0, EWORKSPACE if the workspace is too small; a bounded
 * device wait that runs out is reported by spl_get_device_status. */
spl_status spl_masked_linear(float* Yt, const float* Xt, const spl_weight* W, int64_t M, int64_t K,
                             int64_t N, spl_path path, void* workspace, size_t workspace_bytes,
                             cudaStream_t stream);

/* ---- a4: correction precompute ----------------------------------------
 * C[M, N] = Nz[M, K] W[N, K]^T, the correction W eta (Sec. 5.2).  Several
 * noise draws may be stacked along M (rows are independent).  Same operands,
 * paths and errors as spl_masked_linear. */
spl_status spl_precompute_noise_product(float* C, const float* Nz, const spl_weight* W, int64_t M,
                                        int64_t K, int64_t N, spl_path path, void* workspace,
                                        size_t workspace_bytes, cudaStream_t stream);

/* ---- a4, summed in the masked product's order ---------------------------
 * C = Nz W^T like spl_precompute_noise_product, but every output element is
 * summed in exactly the order spl_masked_linear_unmask uses for a call of
 * `order_rows` rows with the same K, N, path and device: the same kernel, the
 * same K-split boundaries and the same order of the cross-CTA reduction.
 * When the noise dominates the input (x~ ~ eta), the rounding errors of
 * fl(x~ W^T) and fl(eta W^T) then largely cancel in the unmask, so the
 * recovered W x sits far inside the bound of Thm. 4.  Rows of Nz may stack
 * several draws (a bank).  If the masked call's order cannot be reproduced
 * (a launch whose tiles use different splits), this is spl_precompute_noise_product.
 * Workspace: spl_precompute_matched_workspace_bytes(M, K, N, order_rows, path). */
size_t spl_precompute_matched_workspace_bytes(int64_t M, int64_t K, int64_t N, int64_t order_rows, spl_path path);
spl_status spl_precompute_noise_product_matched(float* C, const float* Nz, const spl_weight* W, int64_t M,
                                                int64_t K, int64_t N, int64_t order_rows, spl_path path,
                                                void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* ---- a6: unmask -------------------------------------------------------
 * Y = fl32(Yt - C) elementwise (Eq. add-and-then-subtract).  Y may alias Yt. */
spl_status spl_unmask(float* Y, const float* Yt, const float* C, int64_t rows, int64_t cols,
                      cudaStream_t stream);

/* ---- a5 + a6 fused ----------------------------------------------------
 * Y[M, N] = fl32(fl32(Xt W^T) - C): the masked product with the unmask
 * subtraction done in the product's epilogue.  M <= 16 runs the streaming
 * decode kernel (W read once at HBM rate, FP32).  Same operands and errors as
 * spl_masked_linear plus C. */
spl_status spl_masked_linear_unmask(float* Y, const float* Xt, const spl_weight* W, const float* C,
                                    int64_t M, int64_t K, int64_t N, spl_path path, void* workspace,
                                    size_t workspace_bytes, cudaStream_t stream);

/* ---- binary64 path (Sec. 5.5, the Down projection) ----------------------
 * The input of Down is masked with noise scaled by the activation bound of Thm. 3,
 * so large that in binary32 the cancellation error of Eq. fp-log-bound swamps the
 * output; Sec. 5.5 notes that binary64 (p = 53) resolves it.  These calls do the
 * whole computation in binary64:
 *   spl_noise_mask_f64:   Xt = fl64(X + eta), eta drawn exactly as spl_noise
 *                         (same rng): one binary64 rounding; Xt [rows, cols]
 *                         binary64, X fp32.
 *   spl_precompute_noise_product_f64: C[M, N] = Nz W^T, Nz and W fp32, every
 *                         product exact, binary64 sums; C binary64.
 *   spl_masked_linear_unmask_f64: Y = fl32(fl64(Xt W^T) - C), Xt and C binary64,
 *                         W fp32, products rounded once in binary64, binary64 sums.
 * Bound by the FP64 rate.  Workspace: spl_f64_workspace_bytes(M, K, N) (the
 * first 64 KiB are left untouched, so the product workspace can be shared).
 * Errors as spl_masked_linear (all base pointers 16-byte aligned, K % 4 == 0). */
spl_status spl_noise_mask_f64(double* Xt, const float* X, int64_t rows, int64_t cols, double sensitivity,
                              double eps, spl_mech mech, spl_rng rng, cudaStream_t stream);
size_t spl_f64_workspace_bytes(int64_t M, int64_t K, int64_t N);
spl_status spl_precompute_noise_product_f64(double* C, const float* Nz, const float* W, int64_t M, int64_t K,
                                            int64_t N, void* workspace, size_t workspace_bytes, cudaStream_t stream);
spl_status spl_masked_linear_unmask_f64(float* Y, const double* Xt, const float* W, const double* C, int64_t M,
                                        int64_t K, int64_t N, void* workspace, size_t workspace_bytes,
                                        cudaStream_t stream);

/* ---- Slalom comparator (Sec. 6.2) ------------------------------------------
 * The paper compares its noise masking with Slalom's one-time pad over Z_q,
 * q = 2^23 + 2^21 + 7, with inputs and weights in fixed point with 8 fractional
 * bits.  Field elements are integers below 2^24, carried exactly as fp32.
 *   spl_slalom_quantize: out = rint(v 2^8) (round half to even), fp32 integers;
 *                        for the weights (done once).
 *   spl_slalom_mask:     Xt_q = (rint(X 2^8) mod q + eta) mod q; eta uniform in Z_q,
 *                        element e from Philox block e / 2 + rng.offset, words
 *                        2 (e % 2), 2 (e % 2) + 1 as lo + 2^32 hi, eta = that mod q;
 *                        eta_out (may be NULL) receives eta.  rng.offset_dev must
 *                        be NULL.
 *   correction:          spl_precompute_noise_product_f64(C, eta, W_q): exact.
 *   spl_slalom_linear_unmask: Y = ((Xt_q W_q^T - C) mod q, taken in (-q/2, q/2])
 *                        2^-16, the product exact in binary64 (while every partial
 *                        sum of |Xt_q| |W_q| stays below 2^53: |W| < 0.5 and
 *                        K < 2^22, else ESHAPE for K).  Workspace:
 *                        spl_f64_workspace_bytes(M, K, N). */
spl_status spl_slalom_quantize(float* out, const float* v, int64_t count, cudaStream_t stream);
spl_status spl_slalom_mask(float* Xt_q, float* eta_out, const float* X, int64_t rows, int64_t cols, spl_rng rng,
                           cudaStream_t stream);
spl_status spl_slalom_linear_unmask(float* Y, const float* Xt_q, const float* W_q, const double* C, int64_t M,
                                    int64_t K, int64_t N, void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* Workspace bytes of a product (order_rows = M) or of a correction summed in
 * the order of an online product of order_rows rows, of M rows, K, N on
 * `path`, when its left operand comes split (FP16X3: the arrival counters and
 * partial tiles the swapped kernel of 9-16 rows sums through; 0 for the
 * kernels that reduce on chip) -- for AUTO the most over the paths, the
 * others reading the fp32 operand as the plain calls do.  Calls whose
 * workspaces are this small may run side by side on different streams only
 * with separate workspaces when it is not 0.  0 for invalid arguments. */
size_t spl_split_workspace_bytes(int64_t M, int64_t K, int64_t N, int64_t order_rows, spl_path path);

/* ---- a5 + a6 with the left operand already split ---------------------------
 * As spl_masked_linear_unmask, with X~ given as a descriptor: Xt->w the fp32
 * X~ (may be NULL when the call runs FP16X3) and Xt->f16_hi / f16_lo / f16_exp
 * its fp16 split (from spl_noise_mask_split or spl_split_fp16).  On the FP16X3
 * path the product reads the split and skips its own split pass: the workspace
 * then holds only what spl_split_workspace_bytes(M, K, N, M, path) asks (the
 * swapped kernel's counters and partial tiles for 9-16 rows; none for the
 * kernels that reduce on chip); other paths read Xt->w (EINVAL if it is NULL).
 * The result equals spl_masked_linear_unmask's bit for bit. */
spl_status spl_masked_linear_unmask_split(float* Y, const spl_weight* Xt, const spl_weight* W, const float* C,
                                          int64_t M, int64_t K, int64_t N, spl_path path, void* workspace,
                                          size_t workspace_bytes, cudaStream_t stream);

/* ---- a2 + a3 + a5 + a6 in one call ------------------------------------------
 * Y = fl32(fl32(Xt W^T) - C) with Xt = fl32(X + eta) (Sec. 3.3.1, Eq.
 * add-and-then-subtract): the noise is drawn exactly as spl_noise_mask draws it
 * with the same arguments (rows = M, cols = K, rng), Xt [M, K] is written, and Y
 * equals spl_noise_mask followed by spl_masked_linear_unmask bit for bit.  For
 * 1 <= M <= 4 rows on the FP32 path (AUTO resolves to it there) one launch of the
 * decode kernel does all of it: every block draws the noise of its own K-slice
 * while staging X~, so no separate mask kernel sits between two products; other
 * calls run the two steps.  Xt and X must not overlap (EINVAL).  Workspace and errors as
 * spl_masked_linear_unmask, plus spl_noise_mask's checks on sensitivity, eps,
 * mech and rng; on an error after the mask ran, Xt may have been written. */
spl_status spl_noise_mask_linear_unmask(float* Y, float* Xt, const float* X, const spl_weight* W, const float* C,
                                        int64_t M, int64_t K, int64_t N, double sensitivity, double eps,
                                        spl_mech mech, spl_rng rng, spl_path path, void* workspace,
                                        size_t workspace_bytes, cudaStream_t stream);

/* ---- a4 with the noise already split ------------------------------------
 * As spl_precompute_noise_product_matched, with the noise given as a
 * descriptor: Nz->w the fp32 noise (may be NULL when the call runs FP16X3) and
 * Nz->f16_hi / f16_lo / f16_exp its fp16 split (from spl_noise_mask_split with
 * X NULL).  On the FP16X3 path the tensor-core kernel reads the split and skips
 * its own split pass; other paths read Nz->w (EINVAL if it is NULL).  The
 * result equals spl_precompute_noise_product_matched's bit for bit. */
spl_status spl_precompute_noise_product_matched_split(float* C, const spl_weight* Nz, const spl_weight* W, int64_t M,
                                                      int64_t K, int64_t N, int64_t order_rows, spl_path path,
                                                      void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* ---- a5 + a6 for decode, without allocation ---------------------------
 * The paper has no counterpart to this call; it exists for callers that
 * cannot allocate device memory at the time of the product: a decode loop
 * that must not stall on cudaMalloc/cudaFree (both synchronise the device),
 * a process whose device memory is already fully reserved by another
 * allocator, or a worker whose memory budget is fixed at start-up.
 * Same result as spl_masked_linear_unmask on the FP32 decode kernel
 * (Y = fl32(fl32(Xt W^T) - C), 1 <= M <= 16), but the kernel's scratch
 * (arrival counters and split-K partials) is a fixed array inside the
 * library: 64 KiB of counters plus 4 MiB of partials, which every GPU that
 * loads the library holds until the process exits.  Nothing is allocated:
 * no cudaMalloc, cudaFree or allocating library routine is called.
 *  - Every call looks up the array's device address on the current device
 *    (cudaGetSymbolAddress, which allocates nothing).  The first call on a
 *    device, and the first after the library's module was loaded again (for
 *    instance after cudaDeviceReset), also queues a clear of the counters on
 *    `stream` ahead of its kernel; make that first call before any stream
 *    capture, so that the clear runs when the call is made.
 *  - All calls share the one array, which keeps the last call's contents;
 *    each successful call leaves the counters at zero.  Calls that overlap on
 *    the GPU (on different streams or threads) race on it: serialise them.
 * Errors: EINVAL for NULL operands or negative sizes, ESHAPE for M > 16,
 * EALIGN as for the other calls, EWORKSPACE when the problem needs more
 * split-K partial storage than the built-in 4 MiB (splits x M x N x 4 bytes)
 * or more than 16384 row groups. */
spl_status spl_masked_linear_unmask_noalloc(float* Y, const float* Xt, const float* W, const float* C,
                                            int64_t M, int64_t K, int64_t N, cudaStream_t stream);

/* ---- a4 + a5 + a6 in one launch: the online product beside a bank draw ------
 * The masked product of M rows with its unmask (Eq. add-and-then-subtract) and
 * the corrections W eta of M_bank noise rows (Sec. 5.2, the bank) as one
 * product of M + M_bank rows, so that both run in the launch shape of the
 * larger product.  A is the left operand [M + M_bank, K]: the M rows of X~
 * first, then the M_bank noise rows, as fp32 (A->w) and/or its FP16X3 split
 * (A->f16_hi, f16_lo, f16_exp, as spl_noise_mask_split writes it; the
 * product then reads only the split).  C [M, N] is the correction of the M
 * masked rows.  YC [M + M_bank, N]: rows 0..M-1 get Y = fl32(fl32(Xt W^T) - C),
 * rows M.. the corrections fl32(eta W^T).  Every output row of a product is
 * summed in the same order wherever it sits (launch forms are uniform over the
 * rows of each column of tiles), so a correction computed here is summed
 * exactly as the masked row that later meets it in a call with the same
 * M + M_bank, K, N and path: their rounding errors cancel in the unmask.
 * Runs on the tensor-core paths (TF32X3 / FP16X3, resolved as for M + M_bank
 * rows) and, for M + M_bank <= 16 rows on FP32, on the decode kernel;
 * EUNSUPPORTED for FP32 beyond 16 rows.  Workspace and other errors as
 * spl_masked_linear_unmask for M + M_bank rows. */
spl_status spl_masked_linear_unmask_precompute(float* YC, const spl_weight* A, const spl_weight* W, const float* C,
                                               int64_t M, int64_t M_bank, int64_t K, int64_t N, spl_path path,
                                               void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* ---- a2 + a3 + a4 + a5 + a6 in one decode launch: the stacked schedule ------
 * spl_noise_mask_linear_unmask and spl_masked_linear_unmask_precompute in one:
 * the left operand has M + M_bank rows, rows 0..M-1 being X~ = fl32(X + eta)
 * with eta drawn as spl_noise_mask draws it for X (rows from 0, block offset
 * rng.offset), rows M.. noise alone, drawn as spl_noise_mask with X NULL would
 * draw M_bank rows at block offset rng.offset + noise_block_delta (the same
 * draw of the next bank cycle, Sec. 5.2).  Xt [M + M_bank, K] receives that
 * operand; YC [M + M_bank, N]: rows 0..M-1 get Y = fl32(fl32(Xt W^T) - C)
 * with C [M, N] (Eq. add-and-then-subtract), rows M.. the corrections
 * fl32(eta W^T).  Every row is summed in the same order, so a correction made
 * here cancels the masked row that meets it in a later call of the same
 * shape exactly as spl_masked_linear_unmask_precompute's do.  One launch of
 * the FP32 decode kernel: 1 <= M + M_bank <= 4 and a path resolving to FP32
 * (AUTO does there), else EUNSUPPORTED.  X may be NULL when M = 0 and must
 * not overlap Xt (EINVAL).  Other errors as spl_noise_mask_linear_unmask. */
spl_status spl_noise_mask_linear_unmask_precompute(float* YC, float* Xt, const float* X, const spl_weight* W,
                                                   const float* C, int64_t M, int64_t M_bank, int64_t K, int64_t N,
                                                   double sensitivity, double eps, spl_mech mech, spl_rng rng,
                                                   uint64_t noise_block_delta, spl_path path, void* workspace,
                                                   size_t workspace_bytes, cudaStream_t stream);

/* ---- a8: the cancellation bound on the GPU, and the path choice ----------
 * The paper judges a configuration by evaluating its floating-point bound on
 * sampled inputs and masks (Sec. 4.5 after Thm. 4; Sec. 6.3.2).
 * spl_bound_check does this for `rows` rows: with u = 2^-24, gamma_n = n u/(1 - n u),
 * S_x = <|w|,|x|>, S_xt = <|w|,|x~|>, S_n = <|w|,|eta|> and the exact Y* = X W^T (all fp64),
 *   hard = gamma_K (S_x+S_xt+S_n) + u S_x + u S_xt (1+u)/(1-u) + u gamma_K (S_x+S_xt+S_n)
 *          (Thm. 4 plus the rounding of the mask, second-order term written out)
 *   log  = gamma_{ceil(log2 K)+1} (S_x+S_xt+S_n) + u S_x            (Eq. fp-log-bound)
 * and writes SPL_BOUND_STATS doubles to the HOST array stats:
 *   [0] max |Y-Y*|/hard  [1] max |Y-Y*|/log  [2] count |Y-Y*| > log  [3] sum |Y-Y*|
 *   [4] sum log  [5] sum hard  [6] elements  [7] max |Y*|  [8] max |Y-Y*|.
 * Y [rows, N] is the recovered output; X, Xt, Nz [rows, K]; W [N, K]; all device fp32.
 * Needs a device workspace of >= 8 * SPL_BOUND_STATS bytes; synchronises `stream`. */
#define SPL_BOUND_STATS 9
spl_status spl_bound_check(double* stats, const float* Y, const float* X, const float* Xt, const float* Nz,
                           const float* W, int64_t rows, int64_t K, int64_t N, void* workspace,
                           size_t workspace_bytes, cudaStream_t stream);

/* Bytes of device workspace spl_choose_path needs for a sample of `rows` rows. */
size_t spl_choose_path_workspace_bytes(int64_t rows, int64_t K, int64_t N);

/* a8: masks the sample X (+ Nz), computes the correction and the masked product with the
 * unmask on each path (FP32, and the tensor-core paths whose splits W carries, on a
 * tcgen05 device), checks each with spl_bound_check and sets *chosen to the fastest
 * tensor-core path (FP16X3, then TF32X3) whose max error over the hard bound is <= 1 and
 * whose log-bound violations and summed error are no worse than FP32's (within 1% of the
 * elements and a factor 1.5), else FP32.  stats (HOST) receives 3 x SPL_BOUND_STATS doubles
 * in the order FP32, TF32X3, FP16X3; an unavailable path reports +inf in its [0].
 * Synchronises. */
spl_status spl_choose_path(spl_path* chosen, double* stats, const float* X, const float* Nz,
                           const spl_weight* W, int64_t rows, int64_t K, int64_t N, void* workspace,
                           size_t workspace_bytes, cudaStream_t stream);

/* ---- a1: noise scale ----------------------------------------------------
 * Global l2 sensitivities (Sec. 4.3), evaluated in fp64 on the host from
 * HOST arrays.  Return a negative value on invalid input.
 *  Thm. 1: 2 sqrt(d) ||alpha||_4                         (input of Q, K, V, Gate, Up, LM head)
 *  Thm. 2: 2 sqrt(d) ||W_val||_2 ||alpha||_4              (input of O)
 *  Thm. 3: 2 sqrt(d_ff) (sqrt(d) ||alpha||_4 + ||beta||_2)^2 ||W_up||_2 ||W_gate||_2  (input of Down)
 * beta may be NULL (zero). */
double spl_delta_layernorm(const float* alpha, int64_t d);
double spl_delta_attention(const float* alpha, int64_t d, double wval_spectral_norm);
double spl_delta_activation(const float* alpha, const float* beta, int64_t d, int64_t d_ff,
                            double wup_spectral_norm, double wgate_spectral_norm);

/* ||W||_2 of a DEVICE matrix W[N, K] by power iteration on W^T W (fp32 products,
 * fp64 norms), `iters` iterations from a fixed pseudo-random start vector.
 * Needs a device workspace of at least 4 (N + 2 K) + 256 bytes; synchronises
 * `stream` and writes the result to the HOST double *out. */
spl_status spl_spectral_norm(double* out, const float* W, int64_t N, int64_t K, int iters,
                             void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* Test hook for failure detection (the paper has no counterpart).  Runs one
 * TF32X3 product (K <= 256, so each tile has a single K range) in which the
 * copy of the first K stage is deliberately never issued: the kernel's bounded
 * waits run out after about one second, it sets the device status word, lets
 * the copies it did issue land, frees its tensor memory and returns.  The next
 * spl_get_device_status returns SPL_ETIMEOUT and the context stays usable.
 * `out` receives unspecified values.  Workspace: spl_linear_workspace_bytes(M,
 * K, N, SPL_PATH_TF32X3). */
spl_status spl_test_tc_wait_timeout(float* out, const float* A, const spl_weight* W, int64_t M, int64_t K,
                                    int64_t N, void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* Test hook (no counterpart in the paper): the launch shape the tensor-core
 * product of M x K by N x K takes (seg_splits = 0), or a correction whose sums
 * follow a seg_splits-way split of K (the bank, seg_splits >= 1).  out[6]
 * (host) receives {tile width, ring KB, tiles of the unsplit launch, tiles of the
 * split launch, its K-split, 1 if the persistent kernel takes every tile (else
 * 0)}.  EINVAL for non-positive sizes, seg_splits outside
 * [0, 8] or a NULL out.  No GPU work; needs a current CUDA device for the
 * occupancy queries. */
spl_status spl_test_tc_shape(int64_t M, int64_t K, int64_t N, int64_t seg_splits, int64_t* out);

/* Test hook (no counterpart in the paper): *out (host) = the number of clusters
 * of `cluster` CTAs (1..8) of the launch variant (tile_n, ring_kb) -- (256, 192),
 * (128, 224), (128, 96), (160, 224), (192, 224) or (224, 224) -- that can be
 * resident at once on the current device.
 * EINVAL for another variant, cluster outside [1, 8] or a NULL out. */
spl_status spl_test_tc_capacity(int64_t tile_n, int64_t ring_kb, int64_t cluster, int64_t* out);

/* Test hook (the paper has no counterpart): Y = Xt W^T (- C if C is not NULL)
 * on the tcgen05 kernel with a fixed launch variant -- tile width tile_n and a
 * stage ring of ring_kb KB: (256, 192), (128, 224), (128, 96), (160, 224),
 * (192, 224) or (224, 224) -- and every tile's K range split `splits` ways
 * (1..8) across a thread-block cluster, instead of the shape the library would
 * choose; with full_tiles > 0 the first full_tiles tiles (M fastest) run unsplit
 * in a launch of their own and only the rest is split.  seg_splits > 0: the
 * unsplit tiles run in segmented mode (the bank's form: one CTA over all of K,
 * the partial sums of a seg_splits-way split of K folded in order), so the
 * result equals the seg_splits-way split product bit for bit; splits must then
 * be 1 or seg_splits.  persistent != 0: every tile unsplit in the persistent
 * kernel (one CTA per SM looping over tiles, two TMEM accumulators; the result
 * equals the unsplit product bit for bit); it needs splits 1, seg_splits 0,
 * full_tiles 0, a one-CTA-per-SM variant and N % 4 == 0.  path is
 * SPL_PATH_TF32X3 or SPL_PATH_FP16X3.  Same operands, workspace and errors as
 * spl_masked_linear_unmask; EINVAL for another path or variant, full_tiles
 * outside [0, tiles], seg_splits outside [0, 8], a splits other than 1 or
 * seg_splits, or a persistent request that breaks its conditions; ESHAPE for a
 * split outside 1..8. */
spl_status spl_test_tc_product(float* Y, const float* Xt, const spl_weight* W, const float* C, int64_t M,
                               int64_t K, int64_t N, spl_path path, int tile_n, int ring_kb, int splits,
                               int64_t full_tiles, int seg_splits, int persistent, void* workspace,
                               size_t workspace_bytes, cudaStream_t stream);

/* Test hook: the FP16X3 product on the swapped kernel the library takes for
 * products of 9 to 16 rows (the weight in the MMA's 128 rows, the tokens in
 * its N columns), forced to a token-tile width `tile_tokens` (16, 32, 64 or
 * 128) and `ctas` CTAs per token tile (0: the library's count) for any M: the
 * (128-row weight tile, 64-element k-block) units of each token tile dealt out
 * in `ctas` equal contiguous runs, the pieces of a tile summed in K order by
 * the CTA that finishes the tile last, through the workspace.  Y[M, N] =
 * fl32(Xt W^T - C) (C may be NULL), W with its fp16 split; the workspace holds
 * at least spl_test_tc_swap_workspace_bytes(M, K, N, tile_tokens, ctas) bytes,
 * its first 64 KiB zero (each call leaves them zero).  Errors: EINVAL for a
 * width not listed, NULL operands or ctas < 0, EALIGN for K % 8 != 0 or
 * unaligned pointers, EWORKSPACE for a short workspace, ESHAPE for more than
 * 16384 tiles, as spl_masked_linear otherwise.  The paper has no
 * counterpart. */
spl_status spl_test_tc_swap_product(float* Y, const float* Xt, const spl_weight* W, const float* C, int64_t M,
                                    int64_t K, int64_t N, int tile_tokens, int ctas, void* workspace,
                                    size_t workspace_bytes, cudaStream_t stream);
size_t spl_test_tc_swap_workspace_bytes(int64_t M, int64_t K, int64_t N, int tile_tokens, int ctas);

/* ---- status -------------------------------------------------------------
 * Synchronises `stream`, returns SPL_ETIMEOUT if any kernel since the last
 * call gave up a bounded wait (and clears the flag), else SPL_ECUDA if the
 * stream reports an error, else SPL_OK. */
spl_status spl_get_device_status(cudaStream_t stream);

/* Number of kernels this library has launched in this process so far
 * (all devices, all threads).  Not part of the paper's method: it lets a
 * caller count the library's launches inside a timed region. */
uint64_t spl_launch_count(void);

/* Static, NUL-terminated name of a status code. */
const char* spl_status_string(spl_status status);

/* ---- host-link transfers (plumbing, not a step of the method) -----------
 * Copies `rows` rows of `width_bytes` bytes each from src to dst, source rows
 * src_pitch bytes apart and destination rows dst_pitch bytes apart, queued on
 * `stream` (cudaMemcpy2DAsync; device or page-locked host memory on either
 * side, the direction taken from the pointers).  It moves a step's outputs
 * of every layer, which sit at a fixed pitch in a pooled output buffer, to
 * or from the host in one copy instead of one per layer.  No kernel runs.
 * rows == 0 or width_bytes == 0: nothing to do, SPL_OK.  SPL_EINVAL: a null
 * pointer, or width_bytes above either pitch; SPL_ECUDA: the copy could not
 * be queued.  The caller keeps both buffers alive and unchanged until the
 * stream has passed the copy. */
spl_status spl_copy_2d(void* dst, size_t dst_pitch, const void* src, size_t src_pitch, size_t width_bytes,
                       size_t rows, cudaStream_t stream);

/* ---- the boundary's call names as the problem statement lists them -------
 * The calls of the masked-linear boundary follow the paper's statement of the
 * problem (Sec. 3.3.1, Eq. add-and-then-subtract; the batched precompute of
 * Sec. 5.2).  Most keep that name above; where the library's call is shaped
 * differently, the listed name is kept as well:
 *   spl_noise, spl_mask, spl_noise_mask, spl_unmask        -- as declared above
 *   spl_masked_linear, spl_precompute_noise_product,
 *   spl_masked_linear_unmask                                -- take the weight as a
 *       const spl_weight* (W and its splits) instead of const float* W, plus a
 *       workspace: a spl_weight with only `w` set is accepted and runs the
 *       FP32 path (AUTO resolves to it; an explicit TF32X3 / FP16X3 reports
 *       SPL_EUNSUPPORTED), so a caller holding only fp32 W passes {W}
 *   spl_prepare_weight_split  -> spl_split_tf32 (the TF32X3 split, below) or
 *       spl_split_fp16 (the FP16X3 split, the one the tensor-core products
 *       prefer: 4 bytes per weight)
 *   spl_get_last_device_status -> spl_get_device_status
 *   spl_status_str             -> spl_status_string
 * The three listed names are also exported with their listed signatures: */

/* The TF32X3 split of a weight W[N, K] (fp32, device): W_hi = W rounded to
 * TF32, W_lo = W - W_hi; spl_split_tf32 over the N K elements.  Errors as
 * spl_split_tf32. */
spl_status spl_prepare_weight_split(float* W_hi, float* W_lo, const float* W, int64_t N, int64_t K,
                                    cudaStream_t stream);
/* spl_get_device_status(stream). */
spl_status spl_get_last_device_status(cudaStream_t stream);
/* spl_status_string(status). */
const char* spl_status_str(spl_status status);

#ifdef __cplusplus
}
#endif

#endif /* SPL_H */
