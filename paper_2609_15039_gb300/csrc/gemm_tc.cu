// Split-precision products on the 5th-generation tensor cores (tcgen05, sm_103a):
//   out[M, N] = A[M, K] W[N, K]^T (- C)
// Every operand is split into a high part and a residual, a = a_hi + a_lo, and
// three products per term are accumulated in fp32 (the a_lo w_lo term is dropped):
//   a w ~ a_lo w_hi + a_hi w_lo + a_hi w_hi.
// Two encodings of the split:
//   TF32X3  hi = a rounded to TF32 (11 significant bits), lo = a - hi kept in fp32;
//           the tensor core truncates lo to TF32: per-term error ~2.5 x 2^-21 |a w|.
//           kind::tf32, K = 8 per instruction, 8 bytes per element.
//   FP16X3  each row is first scaled by a power of two so its largest entry lies in
//           [2^14, 2^15); hi = fp16(a 2^e), lo = fp16(a 2^e - hi) (11 + 11 significant
//           bits).  kind::f16 runs at twice the TF32 rate and the split is 4 bytes per
//           element; the power-of-two scales are undone exactly in the epilogue.  Per-term
//           error about 2^-21 |a w| + 2^-39 max|a_row| |w|: an entry more than ~2^-28
//           below its row's largest falls into fp16's subnormal range, where hi + lo keeps
//           an absolute (not relative) error of 2^-25 in the scaled units.
// For rows of ordinary dynamic range each term is within about 3 x 2^-21 of exact, below
// gamma_K = K 2^-24 for K >= 64, so the masked product r = W x~ (Sec. 5.1) and the
// correction W eta (Sec. 5.2) stay inside the binary32 error model the paper's Thm. 4 is
// built on while running on the tensor pipe.  Rows whose small entries carry the sum
// while their large ones meet tiny weights can push the FP16X3 floor past that bound;
// the bound-based path choice on sampled data (spl_choose_path) then takes TF32X3 (whose
// split keeps fp32's exponent range) or FP32.  W is split once, offline; A is split by a pass before the product
// into the workspace, so TMA lands every operand tile directly.
//
// Kernel shape (one CTA per 128 x BN output tile, 6 warps; BN = 256 with a 192 KB ring and
// one CTA per SM, or BN = 128 with a 96 KB ring and two CTAs per SM, so that one CTA's
// epilogue overlaps the other's mainloop):
//   warp 0      TMA producer: per stage A_hi, A_lo, W_hi, W_lo.
//   warp 1      TMEM allocator and MMA issuer: per stage 3 products per k-step into one
//               fp32 accumulator of BN TMEM columns; tcgen05.commit frees the stage.
//   warps 2-5   epilogue: tcgen05.ld 32 lanes x 32 columns, (FP16X3: descale), stage the
//               tile in shared memory; the K-split CTAs of one tile (a thread-block cluster)
//               sum their staged tiles through distributed shared memory in rank order;
//               subtract C (the fused unmask of Eq. add-and-then-subtract) and store.
// Every mbarrier wait is bounded (about 1 s of globaltimer); on expiry the kernel raises
// the device status word, lets issued copies land (again bounded), frees its TMEM and
// returns.  Role loops run warp-wide (lane 0 issues), so no warp is diverged at a barrier.

#include <algorithm>
#include <cstring>

#include <cuda.h>
#include <cuda_fp16.h>

#include "common.cuh"

namespace spl {

__device__ unsigned int g_device_status = 0u;

cudaError_t read_clear_device_status(unsigned int* word) {
  cudaError_t e = cudaMemcpyFromSymbol(word, g_device_status, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  if (*word != 0u) {
    const unsigned int zero = 0u;
    e = cudaMemcpyToSymbol(g_device_status, &zero, sizeof(zero));
  }
  return e;
}

namespace {

constexpr int BM = 128, THREADS = 192;
constexpr unsigned long long kWaitNs = 1000000000ull;  // 1 s per wait
constexpr unsigned long long kDrainNs = 100000000ull;  // 0.1 s to drain on abort
constexpr int MAX_CLUSTER = 8;                         // split-K CTAs of one output tile (portable cluster)
// Longest accumulation chain in TMEM, in k-blocks (1024 elements of K for FP16X3, 512 for TF32X3).
// tcgen05.mma adds its products into the fp32 accumulator with truncation: measured on GB300 at
// zero noise, the error of one chain grows linearly with its length and is almost all bias toward
// zero (max-norm relative error 3.9e-6 at 1024 elements of K on the FP16X3 split, 3.9e-5 at 9728;
// TF32X3, with half the K per instruction, twice that).  A CTA whose K range is longer is cut
// into segments of this many k-blocks: each segment starts a fresh accumulator and is folded into
// the running sum with a round-to-nearest fp32 add (R = fl(R + P)), so the bias of every chain is
// bounded whatever K is, and the folds' own errors are unbiased.  A fold costs ~0.35 us per CTA.
constexpr int kChainBlocks = 32;
constexpr uint32_t AUX_BYTES = 2048;                   // barriers, TMEM slot, abort flag; column scales at +1024

// ---- instruction descriptors (tcgen05.mma kind::tf32 / kind::f16) ---------------
// D = F32 (bits 4-5 = 1); A and B formats at bits 7-9 and 10-12 (f16: 0, tf32: 2);
// both K-major (bits 15, 16 = 0); N >> 3 at bits 17-22; M >> 4 at bits 24-28.
constexpr uint32_t make_idesc(uint32_t ab_format, int m, int n) {
  return (1u << 4) | (ab_format << 7) | (ab_format << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(m >> 4) << 24);
}
static_assert(make_idesc(2, 128, 256) == 0x08400910u, "tf32 idesc encoding");
static_assert(make_idesc(0, 128, 256) == 0x08400010u, "f16 idesc encoding");

// The two encodings.  Operand rows are 64 bytes (64-byte swizzle) in both: 16 fp32 or
// 32 fp16 elements of K per stage.
struct Tf32x3 {
  static constexpr bool kF16 = false;
  static constexpr int BK = 16, UMMA_K = 8, ESZ = 4;
  static constexpr uint32_t FMT = 2;
};
struct Fp16x3 {
  static constexpr bool kF16 = true;
  static constexpr int BK = 32, UMMA_K = 16, ESZ = 2;
  static constexpr uint32_t FMT = 0;
};
// Shared-memory layout of one configuration: tile width BN and a stage ring of RK KB.
// Stage: [A_hi][A_lo][W_hi][W_lo].  A 192 KB ring keeps the most bytes in flight with one CTA
// per SM; a 96 KB ring lets two CTAs share an SM, one streaming while the other finishes.
template <class Md, int BN, int RK>
struct Cfg {
  static_assert(BN % 32 == 0 && BN >= 128 && BN <= 256, "tile width: whole 32-column TMEM loads, one MMA wide");
  static_assert(RK == 96 || RK == 192 || RK == 224, "ring size");
  static constexpr uint32_t A_HALF = BM * Md::BK * Md::ESZ, B_HALF = BN * Md::BK * Md::ESZ;
  static constexpr uint32_t A_HI = 0, A_LO = A_HALF, W_HI = 2 * A_HALF, W_LO = W_HI + B_HALF;
  static constexpr uint32_t STAGE = W_LO + B_HALF;  // bytes TMA brings per stage
  static constexpr uint32_t RING = RK * 1024;
  static constexpr int STAGES = (int)(RING / STAGE);
  static constexpr int CTAS_PER_SM = RK == 96 ? 2 : 1;
  static constexpr uint32_t SMEM = RING + AUX_BYTES + 1024;  // + alignment slack
  static constexpr int RED_STRIDE = BN + 4;                  // floats per row of the staged accumulator
  static constexpr uint32_t IDESC = make_idesc(Md::FMT, BM, BN);
  // TMEM: the accumulator R at column 0 and, in segmented mode, P at column P_OFF (allocations
  // are powers of two of at least 32 columns).
  static constexpr uint32_t P_OFF = BN <= 128 ? 128u : 256u;
  static constexpr uint32_t TMEM_COLS = P_OFF, TMEM_COLS_SEG = 2u * P_OFF;
  static_assert(A_LO % 1024 == 0 && W_HI % 1024 == 0 && W_LO % 1024 == 0 && STAGE % 1024 == 0,
                "swizzle atoms aligned");
  static_assert(STAGES >= 3 && STAGES <= 8, "ring depth");
  static_assert(SMEM <= 232448, "227 KB of dynamic shared memory per block");
  static_assert((size_t)BM * RED_STRIDE * 4 <= RING, "staging fits in the stage ring");
  static_assert(8 * (2 * STAGES + 4) + 16 <= 1024 && 1024 + 4 * BN <= AUX_BYTES, "aux fits");
  // TMA epilogue (unsplit tiles): the tile as BN / 32 chunks of 128 rows x 32 fp32 (128-byte
  // swizzle), C loaded into them and the result stored from them, in the ring once the MMAs are done
  static constexpr uint32_t EPI_CHUNK = BM * 32 * 4;
  static_assert(BN % 32 == 0 && (BN / 32) * EPI_CHUNK <= RING, "epilogue chunks fit in the ring");
};

// Shared-memory matrix descriptor for a K-major operand tile with the 64-byte swizzle:
// 64-byte rows, 8-row (512-byte) atoms stacked along M/N.  start >> 4 in bits 0-13, leading
// byte offset >> 4 in 16-29 (unused by swizzled K-major layouts; 1), stride byte offset >> 4
// (512) in 32-45, descriptor version 1 at bit 46, base offset 0, SWIZZLE_64B = 4 at 61-63.
__device__ __forceinline__ uint64_t make_sdesc_sw64(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1u << 16;
  d |= (uint64_t)(512u >> 4) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)4u << 61;
  return d;
}

// The same for the 128-byte swizzle: 128-byte rows, 8-row (1024-byte) atoms, SWIZZLE_128B = 2.
__device__ __forceinline__ uint64_t make_sdesc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1u << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// ---- PTX wrappers ----------------------------------------------------------------
__device__ __forceinline__ float pow2f(int e) { return __int_as_float((e + 127) << 23); }  // e in [-126, 127]
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ unsigned long long now_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase of the given parity; false if it gave up (deadline passed or
// another role raised *abort).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned long long budget_ns,
                                          volatile int* abort) {
  if (mbar_try(bar, parity)) return true;
  const unsigned long long deadline = now_ns() + budget_ns;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try(bar, parity)) return true;
    if ((it & 63u) == 0u) {
      if (abort && *abort) return false;
      if (now_ns() > deadline) return false;
    }
  }
}
// L2 eviction policies: weight tiles are streamed (first out), A tiles are re-read by every
// output tile of the row block and the rows of C are wanted again in the epilogue (last out).
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(src)
               : "memory");
}
// Waits until the copies have read their shared memory (the CTA may then exit); their writes to
// global memory complete on their own and are visible to the kernels after this one.
__device__ __forceinline__ void tma_store_commit_wait() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
template <class Md, uint32_t IDESC>
__device__ __forceinline__ void mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  if constexpr (Md::kF16) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(IDESC), "r"(accumulate)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(IDESC), "r"(accumulate)
        : "memory");
  }
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// 32 lanes x 32 columns of 32-bit words: thread t gets lane (base + t), columns col..col+31.
__device__ __forceinline__ void tmem_ld_32x32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
// 32 lanes x 32 columns of 32-bit words back to TMEM (thread t writes lane base + t).
__device__ __forceinline__ void tmem_st_32x32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
// 32 lanes x 16 columns of 32-bit words (thread t gets lane base + t).
__device__ __forceinline__ void tmem_ld_32x16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2::evict_last [%0];" ::"l"(p));
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ float4 ld_cluster_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

struct TcMaps {
  CUtensorMap a_hi, a_lo, w_hi, w_lo;
  CUtensorMap y, c;  // TMA epilogue: the output and C as [M, N] fp32, 32 x 128 boxes, 128-byte swizzle
};

// Rows r0..r1 of the staged tile: the S partial tiles of the cluster summed in rank order (S = 1:
// this CTA's own), minus C, stored.  A thread takes P float4 positions per batch and issues every
// load of the batch -- S partials and C for each -- before it adds anything, about 16 loads in
// flight per thread whatever S is, so the epilogue streams instead of waiting load by load.
template <int S, int BN>
__device__ __forceinline__ void reduce_store(const float* red, int r0, int r1, int64_t m0, int64_t n0, int64_t M,
                                             int64_t N, const float* __restrict__ C, float* __restrict__ out,
                                             int64_t c_rows) {
  constexpr int RS = BN + 4;
  constexpr int P = S >= 8 ? 2 : (S >= 4 ? 4 : 8);
  const bool vec = (N & 3) == 0;
  const uint32_t red_base = smem_u32(red);
  const int total = (r1 - r0) * (BN / 4);
  for (int base = threadIdx.x; base < total; base += THREADS * P) {
    float4 part[P][S], cc[P];
    bool live[P];
#pragma unroll
    for (int u = 0; u < P; ++u) {
      const int idx = base + u * THREADS;
      const int r = r0 + idx / (BN / 4), c = 4 * (idx % (BN / 4));
      const int64_t m = m0 + r, n = n0 + c;
      live[u] = idx < total && m < M && n < N;
      cc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (!live[u]) continue;
      if constexpr (S == 1) {
        part[u][0] = *reinterpret_cast<const float4*>(red + r * RS + c);
      } else {
        const uint32_t off = red_base + (uint32_t)((r * RS + c) * 4);
#pragma unroll
        for (int q = 0; q < S; ++q) part[u][q] = ld_cluster_f4(map_to_rank(off, (uint32_t)q));
      }
      if (C && m < c_rows && vec && n + 4 <= N) cc[u] = __ldcs(reinterpret_cast<const float4*>(C + m * N + n));
    }
#pragma unroll
    for (int u = 0; u < P; ++u) {
      if (!live[u]) continue;
      const int idx = base + u * THREADS;
      const int r = r0 + idx / (BN / 4), c = 4 * (idx % (BN / 4));
      const int64_t m = m0 + r, n = n0 + c;
      float4 v = part[u][0];
#pragma unroll
      for (int q = 1; q < S; ++q)  // summed in rank order
        v = make_float4(__fadd_rn(v.x, part[u][q].x), __fadd_rn(v.y, part[u][q].y), __fadd_rn(v.z, part[u][q].z),
                        __fadd_rn(v.w, part[u][q].w));
      float* o = out + m * N + n;
      const bool has_c = C && m < c_rows;
      if (vec && n + 4 <= N) {
        if (has_c)
          v = make_float4(__fsub_rn(v.x, cc[u].x), __fsub_rn(v.y, cc[u].y), __fsub_rn(v.z, cc[u].z),
                          __fsub_rn(v.w, cc[u].w));
        *reinterpret_cast<float4*>(o) = v;
      } else {
        const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (n + j < N) o[j] = has_c ? __fsub_rn(vv[j], C[m * N + n + j]) : vv[j];
      }
    }
  }
}

// One CTA computes a 128 x BN tile of out over the K range of its split (blockIdx.z).
// The `splits` CTAs of a tile form one thread-block cluster (z dimension); their fp32
// partial tiles are summed through distributed shared memory in cluster-rank order, so
// the result does not depend on timing.  An unsplit tile whose output rows are whole 16-byte
// units ends through TMA instead: C's tile is copied into the idle ring, the epilogue warps
// subtract it in place from the accumulator rows they read out of TMEM, and the tile is
// copied out (same arithmetic, same result as the thread loop).
// Segmented mode (seg_blocks > 0, one CTA per tile over all of K): the K range is cut into
// segments of seg_blocks stages, the same boundaries a K-split of the same problem uses; the
// first segment accumulates into R (TMEM columns 0..BN-1), every later one into P (columns
// P_OFF..P_OFF+BN-1), which the epilogue warps fold into R (R = fl(R + P)) before the next segment
// starts.  Each output is then summed in exactly the order of the split launch -- the partials
// of the splits added in rank order -- while one CTA streams its whole K range.
template <class Md, int BN, int RK>
__global__ void __launch_bounds__(THREADS, Cfg<Md, BN, RK>::CTAS_PER_SM)
tc_gemm_kernel(const __grid_constant__ TcMaps maps, float* __restrict__ out, const float* __restrict__ C,
               const int* __restrict__ a_exp, const int* __restrict__ w_exp, int64_t M, int64_t K, int64_t N,
               int64_t k_per_split, int splits, int tile_base, int m_tiles, int skip_kblock, int seg_blocks,
               int epi_tma, int64_t c_rows) {
  using L = Cfg<Md, BN, RK>;
  constexpr int STAGES = L::STAGES, BK = Md::BK, RED_STRIDE = L::RED_STRIDE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* aux = smem + L::RING;
  uint64_t* bars = reinterpret_cast<uint64_t*>(aux);  // full[S], empty[S], accum, seg, fold, c_load
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(aux + 8 * (2 * STAGES + 4));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(aux + 8 * (2 * STAGES + 4) + 8);
  float* red = reinterpret_cast<float*>(smem);  // [BM][RED_STRIDE] staged accumulator, after the mainloop
  float* col_scale = reinterpret_cast<float*>(aux + 1024);  // [BN] FP16X3: 2^-e of the tile's W rows

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Linear tile id, M fastest: the CTAs that read the same weight tile run side by side and share it in L2.
  const int tile = tile_base + (int)blockIdx.x;
  const int64_t m0 = (int64_t)(tile % m_tiles) * BM, n0 = (int64_t)(tile / m_tiles) * BN;
  const int split = blockIdx.z;
  const int64_t kbeg = (int64_t)split * k_per_split;
  const int64_t kend = std::min<int64_t>(K, kbeg + k_per_split);
  const int nk = kend > kbeg ? (int)ceil_div(kend - kbeg, BK) : 0;

  const uint32_t bar_base = smem_u32(bars);
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (STAGES + s); };
  const uint32_t accum_bar = bar_base + 8u * (2 * STAGES);
  const uint32_t seg_bar = bar_base + 8u * (2 * STAGES + 1);   // segmented: a later segment is in P
  const uint32_t fold_bar = bar_base + 8u * (2 * STAGES + 2);  // segmented: P folded into R
  const uint32_t cload_bar = bar_base + 8u * (2 * STAGES + 3);  // TMA epilogue: the tile of C landed
  // TMA epilogue: unsplit tiles whose output rows are whole 16-byte units (chosen by the host)
  const bool tma_epi = epi_tma != 0 && splits == 1;
  const int seg_len = seg_blocks > 0 ? seg_blocks : nk + 1;    // stages per segment
  const int nseg = seg_blocks > 0 ? (int)ceil_div(nk, seg_blocks) : 1;
  const uint32_t tmem_cols = seg_blocks > 0 ? L::TMEM_COLS_SEG : L::TMEM_COLS;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accum_bar, 1);
    mbar_init(seg_bar, 1);
    mbar_init(fold_bar, 4);  // one arrival per epilogue warp
    mbar_init(cload_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(const_cast<uint32_t*>(tmem_slot)), tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer: A_hi, A_lo, W_hi, W_lo ----------------
    // The weight tiles of the first stages do not depend on the kernel before this one (the split
    // of A, which may still be running under programmatic dependent launch): issue them first,
    // then wait for that kernel's results and issue the A tiles.
    uint32_t issued_mask = 0u, phase_mask = 0u;  // per stage: a load was issued / its parity
    bool ok = true;
    const uint64_t pol_w = l2_evict_first(), pol_a = l2_evict_last();
    const int pre = nk < STAGES ? nk : STAGES;
    for (int kb = 0; kb < pre; ++kb) {  // fresh ring: every stage is free
      if (kb == skip_kblock) continue;  // failure-detection test only: this stage never arrives
      if (lane == 0) {
        const uint32_t st = smem_u32(smem + (size_t)kb * L::STAGE);
        const int kx = (int)(kbeg + (int64_t)kb * BK);
        mbar_expect_tx(full_bar(kb), L::STAGE);
        tma_load_2d(st + L::W_HI, &maps.w_hi, full_bar(kb), kx, (int)n0, pol_w);
        tma_load_2d(st + L::W_LO, &maps.w_lo, full_bar(kb), kx, (int)n0, pol_w);
      }
      issued_mask |= 1u << kb;
    }
    pdl_wait();
    for (int kb = 0; kb < pre; ++kb) {
      if (kb == skip_kblock) continue;
      if (lane == 0) {
        const uint32_t st = smem_u32(smem + (size_t)kb * L::STAGE);
        const int kx = (int)(kbeg + (int64_t)kb * BK);
        tma_load_2d(st + L::A_HI, &maps.a_hi, full_bar(kb), kx, (int)m0, pol_a);
        tma_load_2d(st + L::A_LO, &maps.a_lo, full_bar(kb), kx, (int)m0, pol_a);
      }
    }
    __syncwarp();
    for (int kb = pre; kb < nk; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
      ok = __all_sync(0xffffffffu, mbar_wait(empty_bar(s), ph ^ 1u, kWaitNs, abort_flag));
      if (!ok) break;
      if (kb == skip_kblock) continue;
      if (lane == 0) {
        const uint32_t st = smem_u32(smem + (size_t)s * L::STAGE);
        const int kx = (int)(kbeg + (int64_t)kb * BK);
        mbar_expect_tx(full_bar(s), L::STAGE);
        tma_load_2d(st + L::A_HI, &maps.a_hi, full_bar(s), kx, (int)m0, pol_a);
        tma_load_2d(st + L::A_LO, &maps.a_lo, full_bar(s), kx, (int)m0, pol_a);
        tma_load_2d(st + L::W_HI, &maps.w_hi, full_bar(s), kx, (int)n0, pol_w);
        tma_load_2d(st + L::W_LO, &maps.w_lo, full_bar(s), kx, (int)n0, pol_w);
      }
      __syncwarp();
      issued_mask |= 1u << s;
      phase_mask = (phase_mask & ~(1u << s)) | (ph << s);
    }
    pdl_trigger();  // this CTA's loads are issued: the next kernel may be scheduled
    if (!ok) {
      if (lane == 0) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
      }
      // let copies already issued land before the CTA exits
      for (int s = 0; s < STAGES; ++s)
        if (issued_mask & (1u << s)) mbar_wait(full_bar(s), (phase_mask >> s) & 1u, kDrainNs, nullptr);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    bool ok = true;
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
      const int seg = kb / seg_len, in_seg = kb % seg_len;
      if (in_seg == 0 && seg >= 2) {  // P is free once the previous segment has been folded into R
        ok = __all_sync(0xffffffffu, mbar_wait(fold_bar, (uint32_t)(seg - 2) & 1u, kWaitNs, abort_flag));
        if (!ok) break;
      }
      ok = __all_sync(0xffffffffu, mbar_wait(full_bar(s), ph, kWaitNs, abort_flag));
      if (!ok) break;
      if (lane == 0) {
        tc_fence_after();
        const uint32_t st = smem_u32(smem + (size_t)s * L::STAGE);
        const uint32_t acc = tmem + (seg >= 1 ? L::P_OFF : 0u);
#pragma unroll
        for (int kk = 0; kk < BK / Md::UMMA_K; ++kk) {
          const uint32_t koff = kk * 32u;  // one instruction's K is 32 bytes of the 64-byte swizzled row
          const uint32_t first = (in_seg == 0 && kk == 0) ? 0u : 1u;
          mma<Md, L::IDESC>(acc, make_sdesc_sw64(st + L::A_LO + koff), make_sdesc_sw64(st + L::W_HI + koff), first);
          mma<Md, L::IDESC>(acc, make_sdesc_sw64(st + L::A_HI + koff), make_sdesc_sw64(st + L::W_LO + koff), 1u);
          mma<Md, L::IDESC>(acc, make_sdesc_sw64(st + L::A_HI + koff), make_sdesc_sw64(st + L::W_HI + koff), 1u);
        }
        mma_commit(empty_bar(s));  // stage reusable once these MMAs have read it
        if (seg >= 1 && (in_seg == seg_len - 1 || kb == nk - 1)) mma_commit(seg_bar);  // P complete
      }
      __syncwarp();
    }
    pdl_trigger();
    if (lane == 0) {
      if (!ok) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
      }
      mma_commit(accum_bar);  // MMAs already issued must finish before TMEM is read or released
    }
    __syncwarp();
    if (!ok) mbar_wait(accum_bar, 0u, kDrainNs, nullptr);
  } else {
    // ---------------- warps 2..5: stage the accumulator in shared memory ----------------
    // (the ring is free once the MMAs are done)
    // While the mainloop runs: the column scales of the tile into shared memory, and the rows of
    // C this CTA will subtract into L2, so that the epilogue does not wait on DRAM for them.
    const int t = threadIdx.x - 64;  // 0..127
    if constexpr (Md::kF16)
      for (int j = t; j < BN; j += 128) col_scale[j] = pow2f(-((n0 + j < N) ? __ldg(w_exp + n0 + j) : 0));
    if (C && m0 < c_rows && (N & 3) == 0) {
      const int rows_per_rank = (BM + splits - 1) / splits;
      const int rank = splits > 1 ? (int)cluster_rank() : 0;
      const int r0 = rank * rows_per_rank, r1 = (r0 + rows_per_rank < BM) ? r0 + rows_per_rank : BM;
      const int64_t ncols = std::min<int64_t>(BN, N - n0);
      const int lines = (int)ceil_div(ncols * 4, 128);
      for (int i = t; i < (r1 - r0) * lines; i += 128) {
        const int64_t m = m0 + r0 + i / lines;
        if (m < M && m < c_rows) prefetch_l2(C + m * N + n0 + (int64_t)(i % lines) * 32);
      }
    }
    pdl_wait();  // the row exponents of A come from the kernel before this one
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int r_own = 32 * q + lane;
    const int e_row = (Md::kF16 && m0 + r_own < M) ? __ldg(a_exp + m0 + r_own) : 0;
    epilogue_sync();  // col_scale is complete
    bool ok = true;
    for (int f = 0; f + 1 < nseg; ++f) {  // segmented: fold segment f + 1 (in P) into R
      ok = __all_sync(0xffffffffu, mbar_wait(seg_bar, (uint32_t)f & 1u, kWaitNs * 4, abort_flag));
      if (!ok) break;
      tc_fence_after();
      const uint32_t lane_base = tmem + ((uint32_t)(32 * q) << 16);
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float r[32], p[32];
        tmem_ld_32x32(lane_base + (uint32_t)(32 * c), r);
        tmem_ld_32x32(lane_base + L::P_OFF + (uint32_t)(32 * c), p);
#pragma unroll
        for (int i = 0; i < 32; ++i) r[i] = __fadd_rn(r[i], p[i]);
        tmem_st_32x32(lane_base + (uint32_t)(32 * c), r);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(fold_bar);
    }
    bool have = ok && (nk == 0 || mbar_wait(accum_bar, 0u, kWaitNs * 4, abort_flag));
    have = __all_sync(0xffffffffu, have) && !*abort_flag;
    pdl_trigger();
    if (have && tma_epi) {
      // The MMAs are done with the ring: C's tile comes in by TMA as BN / 32 chunks of 128 rows x
      // 32 columns (128-byte swizzle: the 16-byte unit j of row r sits at unit j ^ (r & 7), so the
      // eight rows a quarter-warp touches hit eight different bank groups); each thread takes its
      // row from TMEM, scales it, subtracts C in place, and TMA stores the chunks (rows and columns
      // past M and N are clipped by the copy).
      tc_fence_after();
      const int r = 32 * q + lane;
      const float sr = pow2f(-e_row);
      // chunks holding columns below N (the copies start inside the tensor)
      const int nchunks = (int)std::min<int64_t>(BN / 32, ceil_div(N - n0, (int64_t)32));
      const bool c_tile = C && m0 < c_rows;  // rows past c_rows subtract nothing (the copy fills them with 0)
      if (c_tile && t == 0) {
        mbar_expect_tx(cload_bar, (uint32_t)nchunks * L::EPI_CHUNK);
        const uint64_t pol_c = l2_evict_first();
        for (int c = 0; c < nchunks; ++c)
          tma_load_2d(smem_u32(smem + (size_t)c * L::EPI_CHUNK), &maps.c, cload_bar, (int)n0 + 32 * c, (int)m0, pol_c);
      }
      bool okc = !c_tile || mbar_wait(cload_bar, 0u, kWaitNs, abort_flag);
      okc = __all_sync(0xffffffffu, okc) && !*abort_flag;
      if (okc) {
#pragma unroll 1
        for (int c = 0; c < nchunks; ++c) {
          float v[32];
          if (nk > 0) {
            tmem_ld_32x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(32 * c), v);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = 0.f;
          }
          if constexpr (Md::kF16) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = (v[i] * sr) * col_scale[32 * c + i];  // exact power-of-two scaling
          }
          float4* row = reinterpret_cast<float4*>(smem + (size_t)c * L::EPI_CHUNK + (size_t)r * 128);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float4 o = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
            float4* dst = row + (j ^ (r & 7));
            if (c_tile) {
              const float4 cc = *dst;
              o = make_float4(__fsub_rn(o.x, cc.x), __fsub_rn(o.y, cc.y), __fsub_rn(o.z, cc.z), __fsub_rn(o.w, cc.w));
            }
            *dst = o;
          }
        }
        fence_proxy_async_smem();  // these writes before the copies that read them
        epilogue_sync();
        if (t == 0) {
          for (int c = 0; c < nchunks; ++c)
            tma_store_2d(&maps.y, smem_u32(smem + (size_t)c * L::EPI_CHUNK), (int)n0 + 32 * c, (int)m0);
          tma_store_commit_wait();
        }
      } else if (lane == 0) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
      }
    } else if (have) {
      tc_fence_after();
      const int r = 32 * q + lane;
      float* row = red + (size_t)r * RED_STRIDE;
      const float sr = pow2f(-e_row);
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        if (nk > 0) {
          tmem_ld_32x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(32 * c), v);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.f;
        }
        if constexpr (Md::kF16) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = (v[i] * sr) * col_scale[32 * c + i];  // exact power-of-two scaling
        }
#pragma unroll
        for (int j = 0; j < 32; j += 4)
          *reinterpret_cast<float4*>(row + 32 * c + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
      }
    } else if (lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_device_status, kStatusTimeout);
    }
  }

  // ---- sum the cluster's partial tiles in rank order, subtract C, store ----
  __syncwarp();
  tc_fence_before();
  if (splits > 1) {
    cluster_sync_all();  // every rank's partial tile is staged
  } else {
    __syncthreads();
  }
  if (!tma_epi) {
    const int rank = splits > 1 ? (int)cluster_rank() : 0;
    const int rows_per_rank = (BM + splits - 1) / splits;
    const int r0 = rank * rows_per_rank, r1 = (r0 + rows_per_rank < BM) ? r0 + rows_per_rank : BM;
    switch (splits) {
      case 1: reduce_store<1, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      case 2: reduce_store<2, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      case 3: reduce_store<3, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      case 4: reduce_store<4, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      case 5: reduce_store<5, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      case 6: reduce_store<6, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      case 7: reduce_store<7, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
      default: reduce_store<8, BN>(red, r0, r1, m0, n0, M, N, C, out, c_rows); break;
    }
  }
  __syncwarp();
  if (splits > 1) {
    cluster_sync_all();  // no CTA leaves while others still read its shared memory
  } else {
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, tmem_cols);
  }
}

// Persistent form for launches of several waves of unsplit tiles: one CTA per SM takes the
// tiles blockIdx.x, blockIdx.x + gridDim.x, ... (M fastest, as above).  The stage ring runs on
// across tiles and TMEM holds two buffers (columns 0 and 256).  Tile i keeps its running sum R in
// buffer i % 2; a K range longer than `chain` k-blocks is cut into segments of `chain`, the first
// accumulated into R and each later one into the other buffer P, which the epilogue warps fold into
// R (R = fl(R + P)) before the MMAs take P again.  After the last fold the epilogue warps finish tile
// i from R (C in, Y out, straight between TMEM rows and global memory) while the MMAs of tile i + 1
// accumulate its first segment into buffer (i + 1) % 2 -- the one tile i used as P -- so each
// tile's epilogue overlaps the next tile's mainloop and only the first prologue and the last
// epilogue are exposed.  Every output element is summed exactly as by tc_gemm_kernel with one K
// range and segments of `chain` k-blocks (the same MMAs in the same order, the same folds, the same
// scaling and subtraction), so the two give the same result bit for bit.  Rows of out and C must be
// whole 16-byte units (the host checks).  Every wait is bounded as in tc_gemm_kernel.
//
// Hand-over: every use of a buffer (as R or as P) ends with one tcgen05.commit on buf_full[b] and
// is released by one arrival of each epilogue warp on buf_free[b] (a P after its fold, an R after
// its tile's epilogue), so the k-th use of buffer b waits for release k - 1 and the epilogue's k-th
// wait on buf_full[b] sees completion k.
template <class Md, int BN, int RK>
__global__ void __launch_bounds__(THREADS, 1)
tc_persistent_kernel(const __grid_constant__ TcMaps maps, float* __restrict__ out, const float* __restrict__ C,
                     const int* __restrict__ a_exp, const int* __restrict__ w_exp, int64_t M, int64_t K, int64_t N,
                     int tiles, int m_tiles, int chain, int64_t c_rows) {
  using L = Cfg<Md, BN, RK>;
  constexpr int STAGES = L::STAGES, BK = Md::BK;
  constexpr uint32_t ACC_COLS = 256;  // column offset of the second accumulator
  static_assert(BN <= (int)ACC_COLS, "two accumulators in 512 TMEM columns");
  static_assert(8 * (2 * STAGES + 5) + 16 <= (int)AUX_BYTES, "aux fits");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* aux = smem + L::RING;
  uint64_t* bars = reinterpret_cast<uint64_t*>(aux);  // full[S], empty[S], buf_full[2], buf_free[2], drain
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(aux + 8 * (2 * STAGES + 5));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(aux + 8 * (2 * STAGES + 5) + 8);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int my_tiles = tiles > (int)blockIdx.x ? (tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int nk = (int)ceil_div(K, BK);
  const int seg_len = chain > 0 && chain < nk ? chain : nk;  // k-blocks per segment
  const int nseg = (int)ceil_div(nk, seg_len);
  const uint32_t bar_base = smem_u32(bars);
  auto full_bar = [&](int st) { return bar_base + 8u * st; };
  auto empty_bar = [&](int st) { return bar_base + 8u * (STAGES + st); };
  auto buf_full = [&](int b) { return bar_base + 8u * (2 * STAGES + b); };
  auto buf_free = [&](int b) { return bar_base + 8u * (2 * STAGES + 2 + b); };
  const uint32_t drain_bar = bar_base + 8u * (2 * STAGES + 4);
  auto tile_origin = [&](int i, int64_t& m0, int64_t& n0) {
    const int tile = (int)blockIdx.x + i * (int)gridDim.x;
    m0 = (int64_t)(tile % m_tiles) * BM;
    n0 = (int64_t)(tile / m_tiles) * BN;
  };

  if (threadIdx.x == 0) {
    for (int st = 0; st < STAGES; ++st) {
      mbar_init(full_bar(st), 1);
      mbar_init(empty_bar(st), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(buf_full(b), 1);
      mbar_init(buf_free(b), 4);  // one arrival per epilogue warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(const_cast<uint32_t*>(tmem_slot)), 2 * ACC_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer: the ring runs on across this CTA's tiles ----------------
    uint32_t issued_mask = 0u, phase_mask = 0u;
    bool ok = true;
    const uint64_t pol_w = l2_evict_first(), pol_a = l2_evict_last();
    pdl_wait();  // A comes from the kernel before this one
    uint32_t it = 0;
    for (int i = 0; i < my_tiles && ok; ++i) {
      int64_t m0, n0;
      tile_origin(i, m0, n0);
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int st = (int)(it % STAGES);
        const uint32_t ph = (it / STAGES) & 1u;
        if (it >= (uint32_t)STAGES) {
          ok = __all_sync(0xffffffffu, mbar_wait(empty_bar(st), ph ^ 1u, kWaitNs, abort_flag));
          if (!ok) break;
        }
        if (lane == 0) {
          const uint32_t sa = smem_u32(smem + (size_t)st * L::STAGE);
          const int kx = kb * BK;
          mbar_expect_tx(full_bar(st), L::STAGE);
          tma_load_2d(sa + L::A_HI, &maps.a_hi, full_bar(st), kx, (int)m0, pol_a);
          tma_load_2d(sa + L::A_LO, &maps.a_lo, full_bar(st), kx, (int)m0, pol_a);
          tma_load_2d(sa + L::W_HI, &maps.w_hi, full_bar(st), kx, (int)n0, pol_w);
          tma_load_2d(sa + L::W_LO, &maps.w_lo, full_bar(st), kx, (int)n0, pol_w);
        }
        __syncwarp();
        issued_mask |= 1u << st;
        phase_mask = (phase_mask & ~(1u << st)) | (ph << st);
      }
    }
    pdl_trigger();
    if (!ok) {
      if (lane == 0) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
      }
      for (int st = 0; st < STAGES; ++st)
        if (issued_mask & (1u << st)) mbar_wait(full_bar(st), (phase_mask >> st) & 1u, kDrainNs, nullptr);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer: tile i's segments into buffers i % 2 (R) and (i + 1) % 2 (P) ------
    bool ok = true;
    uint32_t it = 0;
    uint32_t uses[2] = {0u, 0u};  // uses of each buffer so far
    for (int i = 0; i < my_tiles && ok; ++i) {
      for (int sg = 0; sg < nseg && ok; ++sg) {
        const int b = (i & 1) ^ (sg == 0 ? 0 : 1);
        if (uses[b] >= 1) {  // released by the epilogue: P folded, or R's tile finished
          ok = __all_sync(0xffffffffu, mbar_wait(buf_free(b), (uses[b] - 1u) & 1u, kWaitNs * 4, abort_flag));
          if (!ok) break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + (uint32_t)b * ACC_COLS;
        const int kb0 = sg * seg_len, kb1 = std::min(nk, kb0 + seg_len);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int st = (int)(it % STAGES);
          const uint32_t ph = (it / STAGES) & 1u;
          ok = __all_sync(0xffffffffu, mbar_wait(full_bar(st), ph, kWaitNs, abort_flag));
          if (!ok) break;
          if (lane == 0) {
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + (size_t)st * L::STAGE);
#pragma unroll
            for (int kk = 0; kk < BK / Md::UMMA_K; ++kk) {
              const uint32_t koff = kk * 32u;
              const uint32_t first = (kb == kb0 && kk == 0) ? 0u : 1u;
              mma<Md, L::IDESC>(acc, make_sdesc_sw64(sa + L::A_LO + koff), make_sdesc_sw64(sa + L::W_HI + koff),
                                first);
              mma<Md, L::IDESC>(acc, make_sdesc_sw64(sa + L::A_HI + koff), make_sdesc_sw64(sa + L::W_LO + koff), 1u);
              mma<Md, L::IDESC>(acc, make_sdesc_sw64(sa + L::A_HI + koff), make_sdesc_sw64(sa + L::W_HI + koff), 1u);
            }
            mma_commit(empty_bar(st));
          }
          __syncwarp();
        }
        if (!ok) break;
        if (lane == 0) mma_commit(buf_full(b));  // this segment's sums are complete once these MMAs are
        __syncwarp();
        ++uses[b];
      }
    }
    pdl_trigger();
    if (!ok) {
      if (lane == 0) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
        mma_commit(drain_bar);  // MMAs already issued finish before TMEM is released
      }
      __syncwarp();
      mbar_wait(drain_bar, 0u, kDrainNs, nullptr);
    }
  } else {
    // ---------------- warps 2..5: epilogue of tile i from accumulator i % 2 ----------------
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int r = 32 * q + lane;
    const bool vec_ok = (N & 3) == 0;
    // the rows of C a tile subtracts, into L2 while its mainloop runs (tile i + 1's after tile i)
    auto prefetch_c = [&](int i) {
      if (!C || i >= my_tiles) return;
      int64_t pm0, pn0;
      tile_origin(i, pm0, pn0);
      const int64_t ncols = std::min<int64_t>(BN, N - pn0);
      const int lines = (int)ceil_div(ncols * 4, 128);
      for (int j = threadIdx.x - 64; j < BM * lines; j += 128) {
        const int64_t pm = pm0 + j / lines;
        if (pm < M && pm < c_rows) prefetch_l2(C + pm * N + pn0 + (int64_t)(j % lines) * 32);
      }
    };
    pdl_wait();  // C and the row exponents of A come from before this kernel
    prefetch_c(0);
    bool ok = true;
    uint32_t done[2] = {0u, 0u};  // completions of each buffer consumed so far
    for (int i = 0; i < my_tiles; ++i) {
      const int buf = i & 1, pbuf = buf ^ 1;
      int64_t m0, n0;
      tile_origin(i, m0, n0);
      const int64_t m = m0 + r;
      const float sr = (Md::kF16 && m < M) ? pow2f(-__ldg(a_exp + m)) : 1.0f;
      ok = __all_sync(0xffffffffu, mbar_wait(buf_full(buf), done[buf] & 1u, kWaitNs * 4, abort_flag)) &&
           !*abort_flag;  // the first segment, in R
      if (!ok) break;
      ++done[buf];
      for (int sg = 1; sg < nseg && ok; ++sg) {  // fold each later segment (in P) into R
        ok = __all_sync(0xffffffffu, mbar_wait(buf_full(pbuf), done[pbuf] & 1u, kWaitNs * 4, abort_flag)) &&
             !*abort_flag;
        if (!ok) break;
        ++done[pbuf];
        tc_fence_after();
        const uint32_t lane_base = tmem + ((uint32_t)(32 * q) << 16);
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float rv[32], pv[32];
          tmem_ld_32x32(lane_base + (uint32_t)buf * ACC_COLS + (uint32_t)(32 * c), rv);
          tmem_ld_32x32(lane_base + (uint32_t)pbuf * ACC_COLS + (uint32_t)(32 * c), pv);
#pragma unroll
          for (int j = 0; j < 32; ++j) rv[j] = __fadd_rn(rv[j], pv[j]);
          tmem_st_32x32(lane_base + (uint32_t)buf * ACC_COLS + (uint32_t)(32 * c), rv);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(buf_free(pbuf));
      }
      if (!ok) break;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        const int64_t nc = n0 + 32 * c;
        if (nc >= N) break;  // the same for the whole warp
        float v[32];
        tmem_ld_32x32(tmem + (uint32_t)buf * ACC_COLS + ((uint32_t)(32 * q) << 16) + (uint32_t)(32 * c), v);
        if constexpr (Md::kF16) {
#pragma unroll
          for (int j = 0; j < 32; ++j)  // exact power-of-two scaling, as tc_gemm_kernel's col_scale
            v[j] = (v[j] * sr) * pow2f(-((nc + j < N) ? __ldg(w_exp + nc + j) : 0));
        }
        if (m < M && vec_ok) {
          const bool has_c = C && m < c_rows;
          float4 cc[8];
#pragma unroll
          for (int j = 0; j < 8; ++j)
            cc[j] = (has_c && nc + 4 * j < N) ? __ldcs(reinterpret_cast<const float4*>(C + m * N + nc + 4 * j))
                                              : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (nc + 4 * j >= N) continue;
            float4 o = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
            if (has_c)
              o = make_float4(__fsub_rn(o.x, cc[j].x), __fsub_rn(o.y, cc[j].y), __fsub_rn(o.z, cc[j].z),
                              __fsub_rn(o.w, cc[j].w));
            *reinterpret_cast<float4*>(out + m * N + nc + 4 * j) = o;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(buf_free(buf));
      prefetch_c(i + 1);
    }
    pdl_trigger();
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_device_status, kStatusTimeout);
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * ACC_COLS);
  }
}

// ---- few rows: the weight in the MMA's 128 rows, the tokens in its N ------------------------------
// out[M, N] = A[M, K] W[N, K]^T (- C) on FP16X3 for a few tokens (9 to 16 rows: from 17 rows on the
// 128-row tiles of tc_gemm_kernel were as fast on GB300, and up to 8 rows the FP32 decode kernel is
// the library's choice): D = W A^T, so the weight fills the 128 rows of the MMA and the tokens its N
// columns (TN per token tile, a multiple of 16; tokens past M are the zero rows the copy fills in).
// The weight streams once per token tile -- 4 bytes per weight, the same as the fp32 weight the
// decode kernel reads -- while the MMAs do a small fraction of a full tile's work, so the kernel runs
// near HBM rate where a 128-row tile of tokens would be tensor-bound on mostly empty rows.  With so
// little work per MMA the instructions themselves cost time, so the three products of a term take
// two: the tokens' lo and hi rows sit next to each other in shared memory, one MMA of N = 2 TN
// multiplies W_hi by both (columns 0..TN-1: hi*lo; TN..2TN-1: hi*hi) and a second multiplies W_lo
// by the tokens' hi rows into columns 0..TN-1.  The large hi*hi sums and the small cross terms thus
// accumulate apart (the cross terms' truncation error is ~2^-11 smaller) and are added with
// round-to-nearest when a chain is read out.  Row exponents are undone exactly (the weight's per
// MMA row, the tokens' per column).  K-blocks are 64 elements (128-byte rows, 128-byte swizzle):
// measured on GB300, half as many ring round trips per byte made the 64-byte form 10-30% slower.
//
// Work split (stream-K): the (weight tile, k-block) units of one token tile, tile-major, are dealt
// out in `ctas` contiguous runs of equal length (CTA c takes units [c U / ctas, (c + 1) U / ctas)
// of U), so every CTA streams the same number of weight bytes whatever the number of tiles: no
// partly empty wave and no clusters.  A run crosses tile boundaries: its part of one tile (a piece)
// is summed in chains of at most 1024 elements of K (kChainBlocks of the 32-element unit),
// alternating between two TMEM accumulators so that the epilogue reads one chain while the MMAs
// fill the other; the chains of a piece are added in order with round-to-nearest.  A piece that is
// a whole tile goes straight out.  Otherwise its partial tile (8-64 KB) goes to the workspace and
// the CTA bumps the tile's arrival counter; the CTA that arrives last sums the tile's pieces in K
// order (every CTA's slot, its own included), undoes the row scales, subtracts C, stores, and puts
// the counter back to zero for the next call.  No CTA waits on another.  The decomposition depends
// only on N, K and `ctas`, the same for every token tile and every token column, and an element's
// sum does not depend on the other columns of its MMA, so a bank run with the online product's
// `ctas` at any token-tile width reproduces its sums bit for bit.
constexpr int64_t kSwapMaxM = 16;

// Units of CTA c of `ctas` over `total` units: [run_begin(c), run_begin(c + 1)).
__host__ __device__ __forceinline__ int64_t run_begin(int64_t c, int64_t total, int64_t ctas) {
  return c * total / ctas;
}
// The CTA whose run holds unit u (the largest c with run_begin(c) <= u; ctas <= total).
__host__ __device__ __forceinline__ int64_t run_of(int64_t u, int64_t total, int64_t ctas) {
  return ((u + 1) * ctas - 1) / total;
}

template <int TN>
struct SwapCfg {
  static_assert(TN % 16 == 0 && TN >= 16 && TN <= 128, "MMA N of 2 TN: a multiple of 32 up to 256");
  static constexpr int BK = 64;  // fp16 elements of K per 128-byte swizzled row
  static constexpr uint32_t W_HALF = BM * BK * 2, X_HALF = TN * BK * 2;
  static constexpr uint32_t W_HI = 0, W_LO = W_HALF, X_LO = 2 * W_HALF, X_HI = X_LO + X_HALF;
  static constexpr uint32_t STAGE = X_HI + X_HALF;  // bytes TMA brings per stage
  static constexpr uint32_t RING = 192u * 1024u;    // one CTA per SM
  static constexpr int STAGES = (int)(RING / STAGE) > 12 ? 12 : (int)(RING / STAGE);
  static constexpr uint32_t SMEM = RING + AUX_BYTES + 1024;
  static constexpr uint32_t IDESC_HI = make_idesc(0, BM, 2 * TN);  // W_hi x [x_lo; x_hi]
  static constexpr uint32_t IDESC_LO = make_idesc(0, BM, TN);      // W_lo x x_hi
  static constexpr uint32_t BUF = 2 * TN;                          // columns of one accumulator
  static constexpr uint32_t TMEM_COLS = 4 * TN < 64 ? 64u : (uint32_t)(4 * TN);  // two of them
  static constexpr uint32_t AUX_BARS = 8 * (2 * STAGES + 5);  // full[S], empty[S], buf_full[2], buf_free[2], drain
  static constexpr int64_t CHAIN = kChainBlocks * 32 / BK;    // k-blocks per chain: 1024 elements of K
  static_assert(X_HALF % 1024 == 0 && STAGE % 1024 == 0 && X_LO % 1024 == 0, "swizzle atoms aligned");
  static_assert(STAGES >= 3, "ring depth");
  static_assert(AUX_BARS + 16 <= 1024, "barriers fit");
  static_assert(TMEM_COLS <= 512, "TMEM of the CTA");
  static_assert(SMEM + 1024 <= 233472, "shared memory of the CTA");
};

template <int TN>
__global__ void __launch_bounds__(THREADS, 1)
tc_swap_kernel(const __grid_constant__ TcMaps maps, float* __restrict__ out, const float* __restrict__ C,
               const int* __restrict__ x_exp, const int* __restrict__ w_exp, int64_t M, int64_t K, int64_t N, int ctas,
               int64_t c_rows, float* __restrict__ part, unsigned int* __restrict__ counters) {
  using L = SwapCfg<TN>;
  constexpr int STAGES = L::STAGES, BK = L::BK;
  constexpr int64_t CH = L::CHAIN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* aux = smem + L::RING;
  uint64_t* bars = reinterpret_cast<uint64_t*>(aux);
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(aux + L::AUX_BARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(aux + L::AUX_BARS + 8);
  volatile int* last_flag = reinterpret_cast<volatile int*>(aux + L::AUX_BARS + 12);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t nkb = ceil_div(K, (int64_t)BK);
  const int64_t w_tiles = ceil_div(N, (int64_t)BM);
  const int64_t total = w_tiles * nkb;
  const int64_t c = blockIdx.x, tt = blockIdx.y;
  const int64_t m0 = tt * TN;
  const int64_t u0 = run_begin(c, total, ctas), u1 = run_begin(c + 1, total, ctas);

  const uint32_t bar_base = smem_u32(bars);
  auto full_bar = [&](int st) { return bar_base + 8u * st; };
  auto empty_bar = [&](int st) { return bar_base + 8u * (STAGES + st); };
  auto buf_full = [&](int b) { return bar_base + 8u * (2 * STAGES + b); };      // a chain is in buffer b
  auto buf_free = [&](int b) { return bar_base + 8u * (2 * STAGES + 2 + b); };  // buffer b has been read
  const uint32_t drain_bar = bar_base + 8u * (2 * STAGES + 4);

  if (threadIdx.x == 0) {
    for (int st = 0; st < STAGES; ++st) {
      mbar_init(full_bar(st), 1);
      mbar_init(empty_bar(st), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(buf_full(b), 1);
      mbar_init(buf_free(b), 4);  // one arrival per epilogue warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    *last_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(const_cast<uint32_t*>(tmem_slot)), L::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int n_units = (int)(u1 - u0);

  if (warp == 0) {
    // ---------------- TMA producer: the run's units in order, W_hi, W_lo, X_hi, X_lo ----------------
    uint32_t issued_mask = 0u, phase_mask = 0u;
    bool ok = true;
    const uint64_t pol_w = l2_evict_first(), pol_x = l2_evict_last();
    const int pre = n_units < STAGES ? n_units : STAGES;
    for (int j = 0; j < pre; ++j) {  // the weight does not depend on the kernel before this one
      if (lane == 0) {
        const int64_t u = u0 + j;
        const uint32_t st = smem_u32(smem + (size_t)j * L::STAGE);
        mbar_expect_tx(full_bar(j), L::STAGE);
        tma_load_2d(st + L::W_HI, &maps.w_hi, full_bar(j), (int)((u % nkb) * BK), (int)((u / nkb) * BM), pol_w);
        tma_load_2d(st + L::W_LO, &maps.w_lo, full_bar(j), (int)((u % nkb) * BK), (int)((u / nkb) * BM), pol_w);
      }
      issued_mask |= 1u << j;
    }
    pdl_wait();
    for (int j = 0; j < pre; ++j) {
      if (lane == 0) {
        const int64_t u = u0 + j;
        const uint32_t st = smem_u32(smem + (size_t)j * L::STAGE);
        tma_load_2d(st + L::X_HI, &maps.a_hi, full_bar(j), (int)((u % nkb) * BK), (int)m0, pol_x);
        tma_load_2d(st + L::X_LO, &maps.a_lo, full_bar(j), (int)((u % nkb) * BK), (int)m0, pol_x);
      }
    }
    __syncwarp();
    for (int j = pre; j < n_units; ++j) {
      const int st = j % STAGES;
      const uint32_t ph = (uint32_t)(j / STAGES) & 1u;
      ok = __all_sync(0xffffffffu, mbar_wait(empty_bar(st), ph ^ 1u, kWaitNs, abort_flag));
      if (!ok) break;
      if (lane == 0) {
        const int64_t u = u0 + j;
        const int kx = (int)((u % nkb) * BK), ny = (int)((u / nkb) * BM);
        const uint32_t sa = smem_u32(smem + (size_t)st * L::STAGE);
        mbar_expect_tx(full_bar(st), L::STAGE);
        tma_load_2d(sa + L::W_HI, &maps.w_hi, full_bar(st), kx, ny, pol_w);
        tma_load_2d(sa + L::W_LO, &maps.w_lo, full_bar(st), kx, ny, pol_w);
        tma_load_2d(sa + L::X_HI, &maps.a_hi, full_bar(st), kx, (int)m0, pol_x);
        tma_load_2d(sa + L::X_LO, &maps.a_lo, full_bar(st), kx, (int)m0, pol_x);
      }
      __syncwarp();
      issued_mask |= 1u << st;
      phase_mask = (phase_mask & ~(1u << st)) | (ph << st);
    }
    pdl_trigger();
    if (!ok) {
      if (lane == 0) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
      }
      for (int st = 0; st < STAGES; ++st)
        if (issued_mask & (1u << st)) mbar_wait(full_bar(st), (phase_mask >> st) & 1u, kDrainNs, nullptr);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer: chains of at most CH units, buffers alternating ----------------
    bool ok = true;
    int j = 0, it = 0;  // unit of the run, chain of the run
    for (int64_t u = u0; u < u1 && ok;) {
      const int64_t pe = std::min<int64_t>(u1, (u / nkb + 1) * nkb);  // end of the piece
      for (int64_t s = u; s < pe && ok;) {
        const int64_t se = std::min<int64_t>(pe, s + CH);
        const int b = it & 1;
        if (it >= 2) {  // the epilogue has read this buffer's previous chain
          ok = __all_sync(0xffffffffu, mbar_wait(buf_free(b), (uint32_t)((it >> 1) - 1) & 1u, kWaitNs, abort_flag));
          if (!ok) break;
        }
        const uint32_t acc = tmem + (uint32_t)b * L::BUF;
        for (int64_t v = s; v < se; ++v, ++j) {
          const int st = j % STAGES;
          const uint32_t ph = (uint32_t)(j / STAGES) & 1u;
          ok = __all_sync(0xffffffffu, mbar_wait(full_bar(st), ph, kWaitNs, abort_flag));
          if (!ok) break;
          if (lane == 0) {
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + (size_t)st * L::STAGE);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              const uint32_t koff = kk * 32u;  // one instruction's K is 32 bytes of the swizzled row
              const uint32_t first = (v == s && kk == 0) ? 0u : 1u;
              // W_hi x [x_lo; x_hi] (2 TN columns: hi*lo, then hi*hi), then W_lo x x_hi into the cross columns
              mma<Fp16x3, L::IDESC_HI>(acc, make_sdesc_sw128(sa + L::W_HI + koff),
                                       make_sdesc_sw128(sa + L::X_LO + koff), first);
              mma<Fp16x3, L::IDESC_LO>(acc, make_sdesc_sw128(sa + L::W_LO + koff),
                                       make_sdesc_sw128(sa + L::X_HI + koff), 1u);
            }
            mma_commit(empty_bar(st));
            if (v == se - 1) mma_commit(buf_full(b));
          }
          __syncwarp();
        }
        ++it;
        s = se;
      }
      u = pe;
    }
    pdl_trigger();
    if (lane == 0) {
      if (!ok) {
        *abort_flag = 1;
        atomicOr(&g_device_status, kStatusTimeout);
      }
      mma_commit(drain_bar);  // issued MMAs finish before TMEM is released
    }
    __syncwarp();
    if (!ok) mbar_wait(drain_bar, 0u, kDrainNs, nullptr);
  } else {
    // ---------------- warps 2..5: chains summed per piece; pieces out or through the workspace -------
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int r = 32 * q + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(32 * q) << 16);
    pdl_wait();  // the tokens' row exponents, C and the counters come from before this kernel
    bool ok = true;
    int it = 0;
    float run[TN];
#pragma unroll
    for (int i = 0; i < TN; ++i) run[i] = 0.f;
    for (int64_t u = u0; u < u1;) {
      const int64_t t = u / nkb;
      const int64_t pe = std::min<int64_t>(u1, (t + 1) * nkb);
      for (int64_t s = u; s < pe;) {
        const int64_t se = std::min<int64_t>(pe, s + CH);
        const int b = it & 1;
        ok = ok && __all_sync(0xffffffffu, mbar_wait(buf_full(b), (uint32_t)(it >> 1) & 1u, kWaitNs * 4, abort_flag));
        if (ok) {
          tc_fence_after();
          const uint32_t base = lane_base + (uint32_t)b * L::BUF;
#pragma unroll
          for (int cc = 0; cc < TN / 16; ++cc) {
            float hh[16], cr[16];
            tmem_ld_32x16(base + (uint32_t)(TN + 16 * cc), hh);  // hi*hi
            tmem_ld_32x16(base + (uint32_t)(16 * cc), cr);       // the cross terms
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float v = __fadd_rn(hh[i], cr[i]);
              run[16 * cc + i] = s == u ? v : __fadd_rn(run[16 * cc + i], v);
            }
          }
          tc_fence_before();
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(buf_free(b));
        ++it;
        s = se;
      }
      // the piece [u, pe) of weight tile t is in run[] (row r of the tile, tokens m0 ..)
      const int64_t n = t * BM + r;
      const bool whole = u == t * nkb && pe == (t + 1) * nkb;
      bool store = whole;
      if (!whole) {
        // partial tiles [BM][TN]: a row's TN sums contiguous, moved as float4
        const int slot = u == u0 ? 0 : 1;  // a run's first piece, or its last
        float4* dst = reinterpret_cast<float4*>(part + ((tt * ctas + c) * 2 + slot) * (int64_t)(TN * BM)) +
                      r * (TN / 4);
        if (ok) {
#pragma unroll
          for (int i = 0; i < TN / 4; ++i)
            __stcg(dst + i, make_float4(run[4 * i], run[4 * i + 1], run[4 * i + 2], run[4 * i + 3]));
        }
        // the epilogue's stores, then one gpu-scope fence and the arrival (release); the last
        // arrival fences again before the epilogue reads the other pieces (acquire)
        epilogue_sync();
        if (threadIdx.x == 64) {
          const int64_t c_first = run_of(t * nkb, total, ctas), c_last = run_of((t + 1) * nkb - 1, total, ctas);
          unsigned int* cnt = counters + tt * w_tiles + t;
          __threadfence();
          const unsigned int prev = atomicAdd(cnt, 1u);
          const int last = prev == (unsigned int)(c_last - c_first);
          if (last) {
            *cnt = 0u;  // every piece has arrived: ready for the next call
            __threadfence();
          }
          *last_flag = last;
        }
        epilogue_sync();
        store = *last_flag != 0;
        if (store) {
          // the tile's pieces in K order; PB pieces' loads in flight at a time
          constexpr int PB = TN <= 16 ? 8 : (TN <= 32 ? 4 : (TN <= 64 ? 2 : 1));
          const int64_t c_first = run_of(t * nkb, total, ctas), c_last = run_of((t + 1) * nkb - 1, total, ctas);
          for (int64_t cq = c_first; cq <= c_last; cq += PB) {
            float4 buf[PB][TN / 4];
#pragma unroll
            for (int bq = 0; bq < PB; ++bq) {
              if (cq + bq <= c_last) {
                const int sq = run_begin(cq + bq, total, ctas) / nkb == t ? 0 : 1;
                const float4* src =
                    reinterpret_cast<const float4*>(part + ((tt * ctas + cq + bq) * 2 + sq) * (int64_t)(TN * BM)) +
                    r * (TN / 4);
#pragma unroll
                for (int i = 0; i < TN / 4; ++i) buf[bq][i] = __ldcg(src + i);
              }
            }
#pragma unroll
            for (int bq = 0; bq < PB; ++bq) {
              if (cq + bq <= c_last) {
                const bool first = cq + bq == c_first;
#pragma unroll
                for (int i = 0; i < TN / 4; ++i) {
                  run[4 * i] = first ? buf[bq][i].x : __fadd_rn(run[4 * i], buf[bq][i].x);
                  run[4 * i + 1] = first ? buf[bq][i].y : __fadd_rn(run[4 * i + 1], buf[bq][i].y);
                  run[4 * i + 2] = first ? buf[bq][i].z : __fadd_rn(run[4 * i + 2], buf[bq][i].z);
                  run[4 * i + 3] = first ? buf[bq][i].w : __fadd_rn(run[4 * i + 3], buf[bq][i].w);
                }
              }
            }
          }
        }
        epilogue_sync();  // last_flag is read before the next piece may set it
      }
      if (store && ok && n < N) {
        const float sw = pow2f(-__ldg(w_exp + n));
#pragma unroll
        for (int cc = 0; cc < TN / 16; ++cc) {  // 16 tokens at a time: their loads in flight together
          float cv[16];
          int ex[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int64_t m = m0 + 16 * cc + i;
            cv[i] = (C && m < c_rows && m < M) ? __ldcs(C + m * N + n) : 0.f;
            ex[i] = m < M ? __ldg(x_exp + m) : 0;
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int64_t m = m0 + 16 * cc + i;
            if (m < M) {
              // exact power-of-two scaling: the weight row's exponent, then the token's
              const float v = (run[16 * cc + i] * sw) * pow2f(-ex[i]);
              out[m * N + n] = (C && m < c_rows) ? __fsub_rn(v, cv[i]) : v;
            }
          }
        }
      }
      u = pe;
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_device_status, kStatusTimeout);
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, L::TMEM_COLS);
  }
}

// ---- host side: tensor maps ------------------------------------------------------
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D map over a row-major [rows, K] matrix of fp32 or fp16 with a box_k x box_rows box.
bool make_map(CUtensorMap* map, const void* base, bool f16, int64_t rows, int64_t K, int box_k, int box_rows,
              CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const int esize = f16 ? 2 : 4;
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)K * esize};
  cuuint32_t box[2] = {(cuuint32_t)box_k, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
                  const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <class Md, int BN, int RK>
bool set_smem_attr() {
  static bool done[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (!done[dev]) {
    if (cudaFuncSetAttribute(tc_gemm_kernel<Md, BN, RK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)Cfg<Md, BN, RK>::SMEM) != cudaSuccess)
      return false;
    done[dev] = true;
  }
  return true;
}

template <class Md, int BN, int RK>
bool set_smem_attr_persistent() {
  static bool done[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (!done[dev]) {
    if (cudaFuncSetAttribute(tc_persistent_kernel<Md, BN, RK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)Cfg<Md, BN, RK>::SMEM) != cudaSuccess)
      return false;
    done[dev] = true;
  }
  return true;
}

template <int TN>
bool set_smem_attr_swap() {
  static bool done[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (!done[dev]) {
    if (cudaFuncSetAttribute(tc_swap_kernel<TN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)SwapCfg<TN>::SMEM) != cudaSuccess)
      return false;
    done[dev] = true;
  }
  return true;
}

// Token-tile widths of the swapped kernel: 16, 32, 64 for the online products, 128 for the banks of
// several draws (more tokens take several token tiles).
constexpr int kSwapWidths = 4;
constexpr int kSwapTn[kSwapWidths] = {16, 32, 64, 128};

int swap_width_index(int64_t tokens) {
  for (int i = 0; i < kSwapWidths; ++i)
    if (tokens <= kSwapTn[i]) return i;
  return kSwapWidths - 1;
}

// The launch variants: tile width, ring size, CTAs per SM, and the cost constants of the
// launch model below.  Cost of one round of co-resident CTAs, in units of K: F + f s + b K / s
// (F: setup, pipeline fill and epilogue of a CTA; f: the cluster reduction per rank; b: the
// mainloop per K element, relative to the 256-wide tile with the 192 KB ring), fitted to a sweep
// of every variant, split and whole-wave form over the eight Llama and Qwen projections at 128,
// 512, 1024, 2048 and 4096 rows on GB300: the shapes it picks (ties going to the earlier variant,
// as below) are within 0.5% of the best measured, on average over the 40 cases.  A k-step of a narrower tile costs almost as much as
// one of a 256-wide tile (b ~ 1 for every width), so the narrower tiles win only where they fill
// a wave that the 256-wide tiles leave part empty (e.g. 512 x 3072 by 3072: 64 tiles of 192
// columns in clusters of 2 instead of 48 of 256).
struct Variant {
  int bn, rk, cps;
  double F, f, b;
};
constexpr int kVariants = 6;
constexpr Variant kVariant[kVariants] = {{256, 192, 1, 500.0, 20.0, 1.0},   {128, 224, 1, 300.0, 20.0, 1.05},
                                         {128, 96, 2, 250.0, 20.0, 0.95},   {160, 224, 1, 250.0, 20.0, 1.05},
                                         {192, 224, 1, 300.0, 20.0, 1.0},   {224, 224, 1, 550.0, 20.0, 0.97}};

// Co-resident clusters of s CTAs of variant v on the current device; clusters must fit inside
// one GPC, so this is not simply (SMs x CTAs per SM) / s.  Both encodings use the same shared
// memory and block shape for a given variant, so one query serves both.  Cached per device.
template <int BN, int RK>
int query_active_clusters(int s) {
  int n = 0;
  if (!set_smem_attr<Tf32x3, BN, RK>()) return 0;
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(1, 1, (unsigned)s);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = Cfg<Tf32x3, BN, RK>::SMEM;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = (unsigned)s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaOccupancyMaxActiveClusters(&n, tc_gemm_kernel<Tf32x3, BN, RK>, &cfg) != cudaSuccess) n = 0;
  cudaGetLastError();
  return n;
}

int max_active_clusters(int v, int s, int sms) {
  static int cache[64][kVariants][MAX_CLUSTER + 1] = {{{0}}};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return std::max(1, sms * kVariant[v].cps / s);
  int& c = cache[dev][v][s];
  if (c == 0) {
    int n = 0;
    switch (v) {
      case 0: n = query_active_clusters<kVariant[0].bn, kVariant[0].rk>(s); break;
      case 1: n = query_active_clusters<kVariant[1].bn, kVariant[1].rk>(s); break;
      case 2: n = query_active_clusters<kVariant[2].bn, kVariant[2].rk>(s); break;
      case 3: n = query_active_clusters<kVariant[3].bn, kVariant[3].rk>(s); break;
      case 4: n = query_active_clusters<kVariant[4].bn, kVariant[4].rk>(s); break;
      default: n = query_active_clusters<kVariant[5].bn, kVariant[5].rk>(s); break;
    }
    c = n > 0 ? n : std::max(1, sms * kVariant[v].cps / s);
  }
  return c;
}

// Launch shape: a variant, then either one launch with every tile's K split s ways over a
// cluster, or whole waves of unsplit tiles followed by the remaining tiles split (so the last
// wave is not mostly idle).  Cost of a launch in units of K: rounds x (F + f s + b K / s), rounds
// counting co-resident CTAs.  At least 256 of K per CTA; ties go to the earlier variant and to
// fewer splits.
struct TcShape {
  int v;
  int64_t full_tiles;  // tiles of the first, unsplit launch (whole waves)
  int64_t rest_tiles;  // tiles of the second launch
  int rest_splits;
  double cost;
  bool persistent = false;  // one launch of tc_persistent_kernel over every tile (unsplit)
};

// Cost of the persistent form: the first prologue and the last epilogue (F) once, then per tile of
// the busiest CTA its mainloop and a small hand-over (kPersistentTile, in units of K).  With it the
// shapes picked over the eight projections at 512 to 4096 rows (persistent, split and whole-wave
// forms all timed) are within 0.16% of the best measured on average; the persistent form saves 4-7%
// on shapes of several waves (e.g. 2048 x 2560 by 19456: 386.5 against 412.8 us).
constexpr double kPersistentTile = 60.0;

double launch_cost(int v, int64_t tiles, int64_t K, int s, int sms) {
  if (tiles <= 0) return 0.0;
  const int64_t capacity = (int64_t)max_active_clusters(v, s, sms) * s;
  const int64_t rounds = ceil_div(tiles * s, capacity);
  return (double)rounds * (kVariant[v].F + kVariant[v].f * s + kVariant[v].b * (double)K / (double)s);
}

TcShape tc_shape_for(int v, int64_t M, int64_t K, int64_t N, int sms) {
  // the persistent epilogue stores whole float4s: output rows of whole 16-byte units (a launch whose
  // pointers are not 16-byte aligned runs the same tiles unsplit in tc_gemm_kernel: the same sums)
  const bool persistent_ok = (N & 3) == 0;
  const int64_t tiles = ceil_div(M, BM) * ceil_div(N, kVariant[v].bn);
  const int max_s = (int)std::max<int64_t>(1, std::min<int64_t>(MAX_CLUSTER, K / 256));
  TcShape best{v, 0, tiles, 1, 1e300};
  for (int s = 1; s <= max_s; ++s) {
    const double c = launch_cost(v, tiles, K, s, sms);
    if (c < best.cost * (1.0 - 1e-9)) best = TcShape{v, 0, tiles, s, c};
  }
  const int64_t wave = max_active_clusters(v, 1, sms);
  // whole waves of unsplit tiles, cut at whole columns of tiles (M is the fast index), so that every
  // output row of a column is summed the same way wherever it sits in M
  const int64_t m_tiles = ceil_div(M, BM);
  const int64_t full = (tiles / wave) * wave / m_tiles * m_tiles, rest = tiles - full;
  if (full > 0 && rest > 0) {
    const double cf = launch_cost(v, full, K, 1, sms);
    for (int s = 1; s <= max_s; ++s) {
      const double c = cf + launch_cost(v, rest, K, s, sms);
      if (c < best.cost * (1.0 - 1e-9)) best = TcShape{v, full, rest, s, c};
    }
  }
  if (persistent_ok && kVariant[v].cps == 1 && tiles > wave) {  // more than one wave of unsplit tiles
    const double c = kVariant[v].F + (double)ceil_div(tiles, wave) * (kVariant[v].b * (double)K + kPersistentTile);
    if (c < best.cost * (1.0 - 1e-9)) {
      best = TcShape{v, 0, tiles, 1, c};
      best.persistent = true;
    }
  }
  return best;
}

// Shape of a correction whose sums must follow a seg_splits-way split of K (the bank): whole
// waves of unsplit tiles that fold the K ranges in TMEM (segmented mode), then the remaining
// tiles with K split seg_splits ways over a cluster, whose rank-order sum is the same fold; or
// every tile segmented.  The cheapest variant and form.
TcShape tc_bank_shape(int64_t M, int64_t K, int64_t N, int seg_splits, int sms) {
  TcShape best{0, 0, 0, 1, 1e300};
  for (int v = 0; v < kVariants; ++v) {
    const int64_t tiles = ceil_div(M, BM) * ceil_div(N, kVariant[v].bn);
    const double c = launch_cost(v, tiles, K, 1, sms);
    if (c < best.cost * (1.0 - 1e-9)) best = TcShape{v, 0, tiles, 1, c};
    if (seg_splits < 2 || seg_splits > MAX_CLUSTER) continue;
    const int64_t wave = max_active_clusters(v, 1, sms);
    const int64_t full = (tiles / wave) * wave, rest = tiles - full;
    if (rest == 0) continue;
    const double c2 = launch_cost(v, full, K, 1, sms) + launch_cost(v, rest, K, seg_splits, sms);
    if (c2 < best.cost * (1.0 - 1e-9)) best = TcShape{v, full, rest, seg_splits, c2};
  }
  return best;
}

TcShape tc_shape(int64_t M, int64_t K, int64_t N, int sms) {
  TcShape best = tc_shape_for(0, M, K, N, sms);
  for (int v = 1; v < kVariants; ++v) {
    const TcShape t = tc_shape_for(v, M, K, N, sms);
    if (t.cost < best.cost * (1.0 - 1e-9)) best = t;
  }
  return best;
}

// Segments of a CTA whose K range is k_range elements: kChainBlocks when the range is longer, else 0
// (one chain).
template <class Md>
int chain_segments(int64_t k_range) {
  return ceil_div(k_range, (int64_t)Md::BK) > kChainBlocks ? kChainBlocks : 0;
}

template <class Md, int BN, int RK>
spl_status launch_tc(const LinearArgs& a, const uint16_t* a_hi, const uint16_t* a_lo, const int* a_exp,
                     TcShape shape, int skip_kblock, int seg_splits) {
  // Every CTA cuts its K range into chains of at most kChainBlocks k-blocks.  A correction in the
  // order of a seg_splits-way split (seg_splits > 0, the bank) reproduces, per tile, what the online
  // product did: an online split of at most kChainBlocks k-blocks per rank is one chain per rank,
  // summed in rank order, which one CTA over all of K reproduces by folding segments cut at the
  // split's boundaries; an unsplit online product (seg_splits = 1) is folded at kChainBlocks; an
  // online split whose ranks fold chains of their own is reproduced by the same cluster split.
  int seg_blocks = 0;  // segments of the unsplit tiles of a seg_splits launch
  if (seg_splits == 1) {
    seg_blocks = chain_segments<Md>(a.K);
  } else if (seg_splits > 1) {
    const int rank_blocks = (int)(round_up(ceil_div(a.K, seg_splits), Md::BK) / Md::BK);
    if (rank_blocks <= kChainBlocks) {
      seg_blocks = rank_blocks;
    } else {  // every tile as the online launch ran it: split seg_splits ways, each rank folding its chains
      shape.rest_tiles += shape.full_tiles;
      shape.full_tiles = 0;
      shape.rest_splits = seg_splits;
    }
  }
  if (!set_smem_attr<Md, BN, RK>()) return SPL_ECUDA;
  TcMaps maps;
  std::memset(&maps, 0, sizeof(maps));
  const bool f16 = Md::kF16;
  const void* whi = f16 ? (const void*)a.w_h16 : (const void*)a.w_hi;
  const void* wlo = f16 ? (const void*)a.w_l16 : (const void*)a.w_lo;
  if (!make_map(&maps.a_hi, a_hi, f16, a.M, a.K, Md::BK, BM, CU_TENSOR_MAP_SWIZZLE_64B) ||
      !make_map(&maps.a_lo, a_lo, f16, a.M, a.K, Md::BK, BM, CU_TENSOR_MAP_SWIZZLE_64B) ||
      !make_map(&maps.w_hi, whi, f16, a.N, a.K, Md::BK, BN, CU_TENSOR_MAP_SWIZZLE_64B) ||
      !make_map(&maps.w_lo, wlo, f16, a.N, a.K, Md::BK, BN, CU_TENSOR_MAP_SWIZZLE_64B))
    return SPL_ECUDA;
  // TMA epilogue for unsplit tiles: needs output rows (and C's) of whole 16-byte units
  int epi_tma = (a.N & 3) == 0 && aligned16(a.out) && (!a.c || aligned16(a.c)) ? 1 : 0;
  if (epi_tma) {
    if (!make_map(&maps.y, a.out, false, a.M, a.N, 32, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        (a.c && a.c_rows > 0 && !make_map(&maps.c, a.c, false, a.c_rows, a.N, 32, BM, CU_TENSOR_MAP_SWIZZLE_128B)))
      return SPL_ECUDA;
  }
  const int m_tiles = (int)ceil_div(a.M, BM);
  if constexpr (Cfg<Md, BN, RK>::CTAS_PER_SM == 1) {
  if (shape.persistent && seg_splits == 0 && skip_kblock < 0 && epi_tma) {
    // one CTA per SM over every tile (the same sums as one unsplit launch of tc_gemm_kernel)
    if (!set_smem_attr_persistent<Md, BN, RK>()) return SPL_ECUDA;
    const int64_t tiles = shape.full_tiles + shape.rest_tiles;
    if (tiles > 0x7fffffffLL) return SPL_ESHAPE;
    const int ctas = (int)std::min<int64_t>(tiles, max_active_clusters(shape.v, 1, device_sm_count()));
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof(cfg));
    cfg.gridDim = dim3((unsigned)ctas, 1, 1);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = Cfg<Md, BN, RK>::SMEM;
    cfg.stream = a.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, tc_persistent_kernel<Md, BN, RK>, maps, a.out, a.c, a_exp,
                                             (const int*)a.w_exp, a.M, a.K, a.N, (int)tiles, m_tiles, kChainBlocks,
                                             a.c_rows);
    note_launches(1);
    return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
  }
  }
  // The first launch follows the split of A under programmatic dependent launch: its CTAs start
  // (barriers, TMEM, weight tiles) while the split finishes.
  bool first = true;
  auto launch = [&](int64_t tiles, int64_t base, int splits, int seg) -> spl_status {
    if (tiles <= 0) return SPL_OK;
    const int64_t kps = round_up(ceil_div(a.K, splits), Md::BK);
    if (seg == 0) seg = chain_segments<Md>(kps);  // chains of at most kChainBlocks within the CTA's range
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof(cfg));
    cfg.gridDim = dim3((unsigned)tiles, 1, (unsigned)splits);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = Cfg<Md, BN, RK>::SMEM;
    cfg.stream = a.stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = (unsigned)splits;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = first ? 2 : 1;
    first = false;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, tc_gemm_kernel<Md, BN, RK>, maps, a.out, a.c, a_exp,
                                             (const int*)a.w_exp, a.M, a.K, a.N, kps, splits, (int)base, m_tiles,
                                             skip_kblock, seg, epi_tma, a.c_rows);
    note_launches(1);
    return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
  };
  // segmented mode: unsplit tiles fold the K ranges in TMEM; tiles split over a cluster (the same
  // K ranges) sum them in rank order, which is the same fold
  spl_status st = launch(shape.full_tiles, 0, 1, seg_blocks);
  if (st != SPL_OK) return st;
  return launch(shape.rest_tiles, shape.full_tiles, shape.rest_splits, shape.rest_splits > 1 ? 0 : seg_blocks);
}

template <class Md>
spl_status launch_variant(const LinearArgs& a, const uint16_t* hi, const uint16_t* lo, const int* a_exp,
                          const TcShape& shape, int skip_kblock, int seg_splits) {
  static_assert(kVariants == 6, "one case per variant");
  switch (shape.v) {
    case 0: return launch_tc<Md, kVariant[0].bn, kVariant[0].rk>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
    case 1: return launch_tc<Md, kVariant[1].bn, kVariant[1].rk>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
    case 2: return launch_tc<Md, kVariant[2].bn, kVariant[2].rk>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
    case 3: return launch_tc<Md, kVariant[3].bn, kVariant[3].rk>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
    case 4: return launch_tc<Md, kVariant[4].bn, kVariant[4].rk>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
    default: return launch_tc<Md, kVariant[5].bn, kVariant[5].rk>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
  }
}

// CTAs per token tile of the swapped kernel.  Measured on GB300 (the eight Llama and Qwen
// projections at 8 and 16 rows): runs of whole tiles are fastest where the weight tiles number
// between 3/4 of the SMs and all of them (one tile per CTA, no partial tiles: Qwen Gate|Up, 152
// tiles); otherwise 3/4 of the SMs beat all of them by 0.3-1.5 us, fewer partial tiles to sum
// outweighing the longer runs, and 1/2 of them lost 1-4 us.  More tiles than SMs: one CTA per SM.
int swap_ctas(int64_t K, int64_t N, int sms) {
  const int64_t w_tiles = ceil_div(N, BM);
  const int64_t total = w_tiles * ceil_div(K, (int64_t)SwapCfg<16>::BK);
  int64_t c = 3 * (int64_t)sms / 4;
  if (w_tiles > sms) c = sms;
  else if (4 * w_tiles >= 3 * (int64_t)sms) c = w_tiles;
  return (int)std::max<int64_t>(1, std::min<int64_t>(c, total));
}

// Workspace of the swapped kernel's partial tiles: two slots per CTA and token tile of width tn.
size_t swap_partial_bytes(int64_t rows, int tn, int ctas) {
  return (size_t)round_up(ceil_div(rows, (int64_t)tn) * ctas * 2 * tn * BM * 4, 256);
}

template <int TN>
spl_status launch_swap_tn(const LinearArgs& a, const uint16_t* x_hi, const uint16_t* x_lo, const int* x_exp, int ctas,
                          float* part, size_t part_bytes) {
  using L = SwapCfg<TN>;
  if (!set_smem_attr_swap<TN>()) return SPL_ECUDA;
  const int64_t t_tiles = ceil_div(a.M, (int64_t)TN), w_tiles = ceil_div(a.N, BM);
  const int64_t total = w_tiles * ceil_div(a.K, (int64_t)L::BK);
  if (t_tiles * w_tiles > kMaxCounters || t_tiles > 65535) return SPL_ESHAPE;
  if (ctas < 1) return SPL_EINVAL;
  if (ctas > total) ctas = (int)total;  // every CTA at least one unit
  if (!a.ws || !part || part_bytes < swap_partial_bytes(a.M, TN, ctas)) return SPL_EWORKSPACE;
  TcMaps maps;
  std::memset(&maps, 0, sizeof(maps));
  if (!make_map(&maps.a_hi, x_hi, true, a.M, a.K, L::BK, TN, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&maps.a_lo, x_lo, true, a.M, a.K, L::BK, TN, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&maps.w_hi, a.w_h16, true, a.N, a.K, L::BK, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&maps.w_lo, a.w_l16, true, a.N, a.K, L::BK, BM, CU_TENSOR_MAP_SWIZZLE_128B))
    return SPL_ECUDA;
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)ctas, (unsigned)t_tiles, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = L::SMEM;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, tc_swap_kernel<TN>, maps, a.out, a.c, x_exp, (const int*)a.w_exp, a.M,
                                           a.K, a.N, ctas, a.c_rows, part, static_cast<unsigned int*>(a.ws));
  note_launches(1);
  return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
}

// The swapped kernel with token-tile width index w and `ctas` CTAs per token tile (FP16X3, split
// of the tokens given); part: the workspace after the counters (and the split of A).
spl_status launch_swap(const LinearArgs& a, const uint16_t* x_hi, const uint16_t* x_lo, const int* x_exp, int w,
                       int ctas, float* part, size_t part_bytes) {
  switch (w) {
    case 0: return launch_swap_tn<16>(a, x_hi, x_lo, x_exp, ctas, part, part_bytes);
    case 1: return launch_swap_tn<32>(a, x_hi, x_lo, x_exp, ctas, part, part_bytes);
    case 2: return launch_swap_tn<64>(a, x_hi, x_lo, x_exp, ctas, part, part_bytes);
    default: return launch_swap_tn<128>(a, x_hi, x_lo, x_exp, ctas, part, part_bytes);
  }
}

// forced_v >= 0: every tile with that variant, the first forced_full tiles unsplit in a launch of their own
// and the rest with K split forced_splits ways (one launch when forced_full is 0).
// seg_splits > 0: segmented mode, one unsplit launch whose sums follow a seg_splits-way split.
// swap_w >= 0: the swapped kernel with that token-tile width index and swap_s CTAs per token tile
// (0: the library's count, which depends on K and N only, so a bank of any width meets the online
// product's runs).
spl_status run_tc_impl(const LinearArgs& a, int skip_kblock, int forced_v, int forced_splits, int seg_splits = 0,
                       int64_t forced_full = 0, bool forced_persistent = false, int swap_w = -1, int swap_s = 0) {
  const int cc = device_cc();
  if (cc != 100 && cc != 103) return SPL_EUNSUPPORTED;
  const bool f16 = a.path == SPL_PATH_FP16X3;
  if (f16) {
    if (!a.w_h16 || !a.w_l16 || !a.w_exp) return SPL_EUNSUPPORTED;
    if ((a.K & 7) != 0) return SPL_EALIGN;  // fp16 rows must be whole 16-byte units
    if (!aligned16(a.w_h16) || !aligned16(a.w_l16)) return SPL_EALIGN;
  } else {
    if (!a.w_hi || !a.w_lo) return SPL_EUNSUPPORTED;
    if (!aligned16(a.w_hi) || !aligned16(a.w_lo)) return SPL_EALIGN;
  }
  const bool presplit = f16 && a.a_h16 && a.a_l16 && a.a_exp;  // the caller passed the split of A
  if (presplit) {
    if (!aligned16(a.a_h16) || !aligned16(a.a_l16)) return SPL_EALIGN;
  } else {
    if (!a.ws || a.ws_bytes < kCounterBytes + tc_asplit_bytes(a.M, a.K, a.path)) return SPL_EWORKSPACE;
    if (!aligned16(a.ws)) return SPL_EALIGN;
  }
  if (a.M > 0x7fffffffLL || a.N > 0x7fffffffLL || a.K > 0x7fffffffLL) return SPL_ESHAPE;
  if (ceil_div(a.M, BM) * ceil_div(a.N, 128) > 0x7fffffffLL || forced_splits > MAX_CLUSTER) return SPL_ESHAPE;
  if (forced_v >= kVariants) return SPL_EINVAL;
  // split A into the workspace: [counters][FP16X3: row exponents][hi][lo] (unless passed in)
  const int* a_exp = nullptr;
  const void* a_hi = nullptr;
  const void* a_lo = nullptr;
  if (presplit) {
    a_exp = a.a_exp;
    a_hi = a.a_h16;
    a_lo = a.a_l16;
  } else {
    char* base = static_cast<char*>(a.ws) + kCounterBytes;
    const int64_t esz = f16 ? 2 : 4;
    int* exps = nullptr;
    if (f16) {
      exps = reinterpret_cast<int*>(base);
      base += round_up(a.M * 4, 256);
    }
    void* hi_ = base;
    void* lo_ = base + round_up(a.M * a.K * esz, 256);
    const spl_status st =
        f16 ? run_split_fp16(static_cast<uint16_t*>(hi_), static_cast<uint16_t*>(lo_), exps, a.a, a.M, a.K, a.stream)
            : run_split_tf32(static_cast<float*>(hi_), static_cast<float*>(lo_), a.a, a.M * a.K, a.stream);
    if (st != SPL_OK) return st;
    a_exp = exps;
    a_hi = hi_;
    a_lo = lo_;
  }
  if (swap_w >= 0) {  // the swapped kernel; its partial tiles after the counters (and the split of A)
    if (!f16) return SPL_EUNSUPPORTED;
    const int ctas = swap_s > 0 ? swap_s : swap_ctas(a.K, a.N, device_sm_count());
    const size_t off = kCounterBytes + (presplit ? 0 : tc_asplit_bytes(a.M, a.K, a.path));
    if (!a.ws || a.ws_bytes < off) return SPL_EWORKSPACE;
    return launch_swap(a, static_cast<const uint16_t*>(a_hi), static_cast<const uint16_t*>(a_lo), a_exp, swap_w, ctas,
                       reinterpret_cast<float*>(static_cast<char*>(a.ws) + off), a.ws_bytes - off);
  }
  TcShape shape;
  if (forced_v >= 0) {
    const int64_t tiles = ceil_div(a.M, BM) * ceil_div(a.N, kVariant[forced_v].bn);
    shape = TcShape{forced_v, forced_full, tiles - forced_full, forced_splits, 0.0};
    shape.persistent = forced_persistent;
  } else if (seg_splits > 0) {
    shape = tc_bank_shape(a.M, a.K, a.N, seg_splits, device_sm_count());
  } else {
    shape = tc_shape(a.M, a.K, a.N, device_sm_count());
  }
  const uint16_t* hi = static_cast<const uint16_t*>(a_hi);
  const uint16_t* lo = static_cast<const uint16_t*>(a_lo);
  return f16 ? launch_variant<Fp16x3>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits)
             : launch_variant<Tf32x3>(a, hi, lo, a_exp, shape, skip_kblock, seg_splits);
}

}  // namespace

size_t tc_asplit_bytes(int64_t M, int64_t K, spl_path path) {
  if (path == SPL_PATH_FP16X3) return (size_t)(round_up(M * 4, 256) + 2 * round_up(M * K * 2, 256));
  if (path == SPL_PATH_TF32X3) return (size_t)(2 * round_up(M * K * 4, 256));
  return 0;
}

bool tc_swapped(int64_t M, spl_path path) { return path == SPL_PATH_FP16X3 && M <= kSwapMaxM; }

Plan plan_tc(int64_t M, int64_t K, int64_t N, int sms, spl_path path) {
  Plan p{};
  p.kernel = kKernelTc;
  if (tc_swapped(M, path)) {
    p.splits = 1;  // runs of k-blocks, partial tiles summed through the workspace
    p.ws_partials = tc_partial_bytes(M, K, N, M, path);
  } else {
    const TcShape t = tc_shape(M, K, N, sms);
    p.splits = t.rest_splits;  // partials are reduced through distributed shared memory
  }
  p.k_per_split = ceil_div(K, p.splits);
  p.ws_asplit = tc_asplit_bytes(M, K, path);
  return p;
}

size_t tc_partial_bytes(int64_t M, int64_t K, int64_t N, int64_t order_rows, spl_path path) {
  if (!tc_swapped(order_rows, path) || M <= 0 || K <= 0 || N <= 0) return 0;
  const int64_t total = ceil_div(N, BM) * ceil_div(K, (int64_t)SwapCfg<16>::BK);
  const int ctas = (int)std::min<int64_t>(swap_ctas(K, N, device_sm_count()), total);
  return swap_partial_bytes(M, kSwapTn[swap_width_index(M)], ctas);
}

spl_status run_tc(const LinearArgs& a, const Plan& p) {
  (void)p;
  if (tc_swapped(a.M, a.path)) return run_tc_impl(a, -1, -1, 0, 0, 0, false, swap_width_index(a.M));
  return run_tc_impl(a, -1, -1, 0);
}

bool tc_uniform_shape(int64_t M, int64_t K, int64_t N, spl_path path, int* variant, int* splits) {
  if (tc_swapped(M, path)) {  // one launch of the swapped kernel
    *variant = -1;
    *splits = 1;
    return true;
  }
  const TcShape t = tc_shape(M, K, N, device_sm_count());
  if (t.full_tiles > 0 && t.rest_tiles > 0) return false;
  *variant = t.v;
  *splits = t.full_tiles > 0 ? 1 : t.rest_splits;
  return true;
}

spl_status run_tc_matched(const LinearArgs& a, int64_t order_rows) {
  if (tc_swapped(order_rows, a.path))  // the swapped kernel with the online runs; a width for all of M
    return run_tc_impl(a, -1, -1, 0, 0, 0, false, swap_width_index(a.M), 0);
  int variant = 0, splits = 1;
  if (!tc_uniform_shape(order_rows, a.K, a.N, a.path, &variant, &splits)) return SPL_EINVAL;
  if (splits < 1 || splits > MAX_CLUSTER) return SPL_ESHAPE;
  return run_tc_impl(a, -1, -1, 0, splits);
}

}  // namespace spl

// Failure-detection test hook: one TF32X3 product in which the copy of the first K stage is
// never issued, so the kernel's bounded waits run out (about 1 s), it raises the device status
// word and returns.  The paper has no counterpart.
extern "C" spl_status spl_test_tc_wait_timeout(float* out, const float* A, const spl_weight* W, int64_t M, int64_t K,
                                               int64_t N, void* workspace, size_t workspace_bytes,
                                               cudaStream_t stream) {
  using namespace spl;
  if (!out || !A || !W || !W->w || !W->tf32_hi || !W->tf32_lo || M <= 0 || N <= 0 || K <= 0 || (K & 3))
    return SPL_EINVAL;
  if (K > 256) return SPL_ESHAPE;  // one K range per tile: the skipped stage belongs to every CTA
  LinearArgs args = make_args(out, A, *W, nullptr, M, K, N, workspace, workspace_bytes, stream, SPL_PATH_TF32X3);
  return run_tc_impl(args, 0, 0, 1);
}

// Test hook: the launch shape the tensor-core product (seg_splits = 0) or a correction in the order
// of a seg_splits-way split (seg_splits > 0) takes: out = {tile width, ring KB, tiles of the
// unsplit launch, tiles of the split launch, its K-split, 1 if the persistent kernel takes every
// tile}.  The paper has no counterpart.
extern "C" spl_status spl_test_tc_shape(int64_t M, int64_t K, int64_t N, int64_t seg_splits, int64_t* out) {
  using namespace spl;
  if (!out || M <= 0 || K <= 0 || N <= 0 || seg_splits < 0 || seg_splits > MAX_CLUSTER) return SPL_EINVAL;
  const int sms = device_sm_count();
  const TcShape t = seg_splits > 0 ? tc_bank_shape(M, K, N, (int)seg_splits, sms) : tc_shape(M, K, N, sms);
  out[0] = kVariant[t.v].bn;
  out[1] = kVariant[t.v].rk;
  out[2] = t.full_tiles;
  out[3] = t.rest_tiles;
  out[4] = t.rest_splits;
  out[5] = t.persistent ? 1 : 0;
  return SPL_OK;
}

// Test hook: co-resident clusters of `cluster` CTAs of the launch variant (tile_n, ring_kb) on the
// current device (the occupancy query the launch shapes are planned with).  The paper has no
// counterpart.
extern "C" spl_status spl_test_tc_capacity(int64_t tile_n, int64_t ring_kb, int64_t cluster, int64_t* out) {
  using namespace spl;
  if (!out || cluster < 1 || cluster > MAX_CLUSTER) return SPL_EINVAL;
  for (int v = 0; v < kVariants; ++v)
    if (kVariant[v].bn == tile_n && kVariant[v].rk == ring_kb) {
      *out = max_active_clusters(v, (int)cluster, device_sm_count());
      return SPL_OK;
    }
  return SPL_EINVAL;
}

// Test hook: the tensor-core product with a fixed tile width and K-split, so that tests cover
// every kernel instance and a sweep can time each launch shape; seg_splits > 0 runs the unsplit
// tiles in segmented mode (the bank's form), their sums following a seg_splits-way split of K;
// persistent != 0 runs every tile unsplit in the persistent kernel.  The paper has no counterpart.
extern "C" spl_status spl_test_tc_product(float* out, const float* A, const spl_weight* W, const float* C, int64_t M,
                                          int64_t K, int64_t N, spl_path path, int tile_n, int ring_kb, int splits,
                                          int64_t full_tiles, int seg_splits, int persistent, void* workspace,
                                          size_t workspace_bytes, cudaStream_t stream) {
  using namespace spl;
  if (!out || !A || !W || !W->w || M <= 0 || N <= 0 || K <= 0) return SPL_EINVAL;
  if (path != SPL_PATH_TF32X3 && path != SPL_PATH_FP16X3) return SPL_EINVAL;
  int v = -1;
  for (int i = 0; i < kVariants; ++i)
    if (kVariant[i].bn == tile_n && kVariant[i].rk == ring_kb) v = i;
  if (v < 0) return SPL_EINVAL;
  if (splits < 1 || splits > MAX_CLUSTER) return SPL_ESHAPE;
  if ((K & 3) != 0) return SPL_EALIGN;
  if (!aligned16(out) || !aligned16(A) || (C && !aligned16(C))) return SPL_EALIGN;
  const int64_t tiles = ceil_div(M, BM) * ceil_div(N, (int64_t)tile_n);
  if (full_tiles < 0 || full_tiles > tiles) return SPL_EINVAL;
  if (seg_splits < 0 || seg_splits > MAX_CLUSTER || (seg_splits > 0 && splits > 1 && splits != seg_splits))
    return SPL_EINVAL;
  if (persistent && (splits != 1 || seg_splits != 0 || full_tiles != 0 || kVariant[v].cps != 1 || (N & 3) != 0))
    return SPL_EINVAL;
  const LinearArgs args = make_args(out, A, *W, C, M, K, N, workspace, workspace_bytes, stream, path);
  return run_tc_impl(args, -1, v, splits, seg_splits, full_tiles, persistent != 0);
}

// Test hook: the swapped tensor-core product (FP16X3, the weight in the MMA's rows, the tokens in its
// columns) with a fixed token-tile width (16, 32, 64 or 128) and `ctas` CTAs per token tile (0: the
// library's count), whatever M is, so that tests cover every kernel instance and compare widths and
// run lengths.  The paper has no counterpart.
extern "C" spl_status spl_test_tc_swap_product(float* out, const float* A, const spl_weight* W, const float* C,
                                               int64_t M, int64_t K, int64_t N, int tile_tokens, int ctas,
                                               void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  using namespace spl;
  if (!out || !A || !W || !W->w || M <= 0 || N <= 0 || K <= 0 || ctas < 0) return SPL_EINVAL;
  int w = -1;
  for (int i = 0; i < kSwapWidths; ++i)
    if (kSwapTn[i] == tile_tokens) w = i;
  if (w < 0) return SPL_EINVAL;
  if ((K & 7) != 0) return SPL_EALIGN;
  if (!aligned16(out) || !aligned16(A) || (C && !aligned16(C))) return SPL_EALIGN;
  const LinearArgs args = make_args(out, A, *W, C, M, K, N, workspace, workspace_bytes, stream, SPL_PATH_FP16X3);
  return run_tc_impl(args, -1, -1, 0, 0, 0, false, w, ctas);
}

// Workspace bytes spl_test_tc_swap_product needs for these arguments: the counters, the split of A
// and the partial tiles.  0 for arguments it refuses.
extern "C" size_t spl_test_tc_swap_workspace_bytes(int64_t M, int64_t K, int64_t N, int tile_tokens, int ctas) {
  using namespace spl;
  if (M <= 0 || K <= 0 || N <= 0 || ctas < 0) return 0;
  bool listed = false;
  for (int i = 0; i < kSwapWidths; ++i) listed = listed || kSwapTn[i] == tile_tokens;
  if (!listed) return 0;
  const int64_t total = ceil_div(N, BM) * ceil_div(K, (int64_t)SwapCfg<16>::BK);
  const int p = (int)std::min<int64_t>(total, ctas > 0 ? ctas : swap_ctas(K, N, device_sm_count()));
  return kCounterBytes + tc_asplit_bytes(M, K, SPL_PATH_FP16X3) + swap_partial_bytes(M, tile_tokens, p);
}
