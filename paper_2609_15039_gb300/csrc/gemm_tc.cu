// Split-precision products on the 5th-generation tensor cores (tcgen05, sm_103a):
//   out[M, N] = A[M, K] W[N, K]^T (- C)
// Every operand is split into a high part and a residual, a = a_hi + a_lo, and
// three products per term are accumulated in fp32 (the a_lo w_lo term is dropped):
//   a w ~ a_lo w_hi + a_hi w_lo + a_hi w_hi.
// Two encodings of the split:
//   TF32X3  hi = a rounded to TF32 (11 significant bits), lo = a - hi kept in fp32;
//           the tensor core truncates lo to TF32: per-term error ~2.5 x 2^-21 |a w|.
//           kind::tf32, K = 8 per instruction; W split offline, 8 bytes per weight.
//   FP16X3  each row is first scaled by a power of two so its largest entry lies in
//           [2^14, 2^15); hi = fp16(a 2^e), lo = fp16(a 2^e - hi) (11 + 11 significant
//           bits); per-term error ~2^-21 |a w|.  kind::f16 runs at twice the TF32 rate
//           and the split is 4 bytes per element; the power-of-two scales are undone
//           exactly in the epilogue.  A is split by a pass before the product (into
//           the workspace), so TMA lands every operand tile directly and the whole
//           ring carries loads in flight.
// Either way each term is within about 3 x 2^-21 of exact, below gamma_K = K 2^-24 for
// K >= 64, so the masked product r = W x~ (Sec. 5.1) and the correction W eta (Sec. 5.2)
// stay inside the binary32 error model the paper's Thm. 4 is built on while running on
// the tensor pipe.
//
// Kernel shape (one CTA per 128 x 256 output tile, one CTA per SM, 6 warps):
//   warp 0      TMA producer: per stage the A tile(s) and W_hi, W_lo.
//   warps 2-5   TF32X3: split the raw fp32 A tile into its hi/lo operand tiles in shared
//               memory during the mainloop.  Both modes: the epilogue.
//   warp 1      TMEM allocator and MMA issuer: per stage 2 k-steps x 3 products into one
//               fp32 accumulator of 256 TMEM columns; tcgen05.commit frees the stage.
//   epilogue    tcgen05.ld 32 lanes x 32 columns, (FP16X3: descale), stage the tile in
//               shared memory; the K-split CTAs of one tile (a thread-block cluster) sum
//               their staged tiles through distributed shared memory in rank order;
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

constexpr int BM = 128, BN = 256, THREADS = 192;
constexpr uint32_t TMEM_COLS = 256;
constexpr unsigned long long kWaitNs = 1000000000ull;  // 1 s per wait
constexpr unsigned long long kDrainNs = 100000000ull;  // 0.1 s to drain on abort
constexpr int MAX_CLUSTER = 8;                         // split-K CTAs of one output tile (portable cluster)
constexpr int RED_STRIDE = BN + 4;                     // floats per row of the staged accumulator
constexpr uint32_t RING_BYTES = 192 * 1024;            // stage ring (both modes)
constexpr uint32_t AUX_BYTES = 2048;                   // barriers, TMEM slot, abort flag, exponents
constexpr uint32_t SMEM_BYTES = RING_BYTES + AUX_BYTES + 1024;  // + alignment slack
static_assert((size_t)BM * RED_STRIDE * 4 <= RING_BYTES, "staging fits in the stage ring");

// ---- instruction descriptors (tcgen05.mma kind::tf32 / kind::f16) ---------------
// D = F32 (bits 4-5 = 1); A and B formats at bits 7-9 and 10-12 (f16: 0, tf32: 2);
// both K-major (bits 15, 16 = 0); N >> 3 at bits 17-22; M >> 4 at bits 24-28.
constexpr uint32_t make_idesc(uint32_t ab_format, int m, int n) {
  return (1u << 4) | (ab_format << 7) | (ab_format << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(m >> 4) << 24);
}
static_assert(make_idesc(2, BM, BN) == 0x08400910u, "tf32 idesc encoding");
static_assert(make_idesc(0, BM, BN) == 0x08400010u, "f16 idesc encoding");

// The two modes.  Stage layout: [A_hi][A_lo][W_hi][W_lo]; in TF32X3 the raw A tile lands in
// the A_hi slot and is split in place by warps 2-5; in FP16X3 TMA brings all four tiles.
// Operand rows are 64 bytes (64-byte swizzle) in both modes: 16 fp32 or 32 fp16 elements of K.
struct Tf32x3 {
  static constexpr bool kF16 = false;
  static constexpr int BK = 16;  // K elements per stage
  static constexpr int STAGES = 4;
  static constexpr int UMMA_K = 8;
  static constexpr uint32_t A_HALF = BM * BK * 4, B_HALF = BN * BK * 4;
  static constexpr uint32_t IDESC = make_idesc(2, BM, BN);
};
struct Fp16x3 {
  static constexpr bool kF16 = true;
  static constexpr int BK = 32;
  static constexpr int STAGES = 4;
  static constexpr int UMMA_K = 16;
  static constexpr uint32_t A_HALF = BM * BK * 2, B_HALF = BN * BK * 2;
  static constexpr uint32_t IDESC = make_idesc(0, BM, BN);
};
template <class Md>
struct Layout {
  static constexpr uint32_t A_HI = 0, A_LO = Md::A_HALF, W_HI = 2 * Md::A_HALF, W_LO = W_HI + Md::B_HALF;
  static constexpr uint32_t STAGE = W_LO + Md::B_HALF;
  static constexpr uint32_t TX = (Md::kF16 ? 2 : 1) * Md::A_HALF + 2 * Md::B_HALF;  // bytes TMA brings
  static_assert(STAGE * Md::STAGES <= RING_BYTES, "ring fits");
  static_assert(A_LO % 1024 == 0 && W_HI % 1024 == 0 && STAGE % 1024 == 0, "swizzle atoms aligned");
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

// ---- PTX wrappers ----------------------------------------------------------------
__device__ __forceinline__ float tf32_rna(float v) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(v));
  return __uint_as_float(r);
}
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
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
template <class Md>
__device__ __forceinline__ void mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  if constexpr (Md::kF16) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(Md::IDESC), "r"(accumulate)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(Md::IDESC), "r"(accumulate)
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
__device__ __forceinline__ void converter_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

struct TcMaps {
  CUtensorMap a, a_lo, w_hi, w_lo;  // TF32X3: a = raw fp32 A (a_lo unused); FP16X3: a = A_hi, a_lo = A_lo
};

// One CTA computes a 128 x 256 tile of out over the K range of its split (blockIdx.z).
// The `splits` CTAs of a tile form one thread-block cluster (z dimension); their fp32
// partial tiles are summed through distributed shared memory in cluster-rank order, so
// the result does not depend on timing.
template <class Md>
__global__ void __launch_bounds__(THREADS, 1)
tc_gemm_kernel(const __grid_constant__ TcMaps maps, float* __restrict__ out, const float* __restrict__ C,
               const int* __restrict__ a_exp, const int* __restrict__ w_exp, int64_t M, int64_t K, int64_t N,
               int64_t k_per_split, int splits, int tile_base, int m_tiles, int skip_kblock) {
  using L = Layout<Md>;
  constexpr int STAGES = Md::STAGES, BK = Md::BK;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* aux = smem + RING_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(aux);  // full[S], conv[S], empty[S], accum
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(aux + 8 * (3 * STAGES + 1));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(aux + 8 * (3 * STAGES + 1) + 8);
  int* ea = reinterpret_cast<int*>(aux + 512);    // [BM]  FP16X3: row exponents of A
  int* ew = reinterpret_cast<int*>(aux + 1024);   // [BN]  FP16X3: row exponents of W (whole rows)
  float* red = reinterpret_cast<float*>(smem);    // [BM][RED_STRIDE] staged accumulator, after the mainloop

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
  auto conv_bar = [&](int s) { return bar_base + 8u * (STAGES + s); };
  auto empty_bar = [&](int s) { return bar_base + 8u * (2 * STAGES + s); };
  const uint32_t accum_bar = bar_base + 8u * (3 * STAGES);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(conv_bar(s), 4);  // one arrival per converter warp
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accum_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(const_cast<uint32_t*>(tmem_slot)), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer: raw A, W_hi, W_lo ----------------
    uint32_t issued_mask = 0u, phase_mask = 0u;  // per stage: a load was issued / its parity
    bool ok = true;
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
      ok = __all_sync(0xffffffffu, mbar_wait(empty_bar(s), ph ^ 1u, kWaitNs, abort_flag));
      if (!ok) break;
      if (kb == skip_kblock) continue;  // failure-detection test only: this stage never arrives
      if (lane == 0) {
        const uint32_t st = smem_u32(smem + (size_t)s * L::STAGE);
        const int kx = (int)(kbeg + (int64_t)kb * BK);
        mbar_expect_tx(full_bar(s), L::TX);
        tma_load_2d(st + L::A_HI, &maps.a, full_bar(s), kx, (int)m0);
        if constexpr (Md::kF16) tma_load_2d(st + L::A_LO, &maps.a_lo, full_bar(s), kx, (int)m0);
        tma_load_2d(st + L::W_HI, &maps.w_hi, full_bar(s), kx, (int)n0);
        tma_load_2d(st + L::W_LO, &maps.w_lo, full_bar(s), kx, (int)n0);
      }
      __syncwarp();
      issued_mask |= 1u << s;
      phase_mask = (phase_mask & ~(1u << s)) | (ph << s);
    }
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
      // FP16X3: the operand tiles are ready when TMA lands them; TF32X3: when A is split
      ok = __all_sync(0xffffffffu, mbar_wait(Md::kF16 ? full_bar(s) : conv_bar(s), ph, kWaitNs, abort_flag));
      if (!ok) break;
      if (lane == 0) {
        tc_fence_after();
        const uint32_t st = smem_u32(smem + (size_t)s * L::STAGE);
#pragma unroll
        for (int kk = 0; kk < BK / Md::UMMA_K; ++kk) {
          const uint32_t koff = kk * 32u;  // one instruction's K is 32 bytes of the 64-byte swizzled row
          const uint32_t first = (kb == 0 && kk == 0) ? 0u : 1u;
          mma<Md>(tmem, make_sdesc_sw64(st + L::A_LO + koff), make_sdesc_sw64(st + L::W_HI + koff), first);
          mma<Md>(tmem, make_sdesc_sw64(st + L::A_HI + koff), make_sdesc_sw64(st + L::W_LO + koff), 1u);
          mma<Md>(tmem, make_sdesc_sw64(st + L::A_HI + koff), make_sdesc_sw64(st + L::W_HI + koff), 1u);
        }
        mma_commit(empty_bar(s));  // stage reusable once these MMAs have read it
      }
      __syncwarp();
    }
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
    // ---------------- warps 2..5: split A during the mainloop, then the epilogue ----------------
    const int t = threadIdx.x - 64;  // 0..127
    if constexpr (Md::kF16) {
      // power-of-two row exponents of A (whole rows, from the exponent pass) and of this tile's W rows
      ea[t] = (m0 + t < M) ? a_exp[m0 + t] : 0;
      for (int j = t; j < BN; j += 128) ew[j] = (n0 + j < N) ? w_exp[n0 + j] : 0;
      converter_sync();
    }
    bool ok = true;
    if constexpr (!Md::kF16) {
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
        ok = mbar_wait(full_bar(s), ph, kWaitNs, abort_flag);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        // The raw tile sits in the hi slot; hi and lo use the same swizzled positions, so the split is
        // elementwise and in place.  Consecutive threads take consecutive 16-byte chunks.
        uint8_t* st = smem + (size_t)s * L::STAGE;
        float4* hi = reinterpret_cast<float4*>(st + L::A_HI);
        float4* lo = reinterpret_cast<float4*>(st + L::A_LO);
#pragma unroll
        for (int j = 0; j < (int)(Md::A_HALF / 16) / 128; ++j) {
          const int i = t + 128 * j;
          const float4 v = hi[i];
          const float4 h = make_float4(tf32_rna(v.x), tf32_rna(v.y), tf32_rna(v.z), tf32_rna(v.w));
          hi[i] = h;
          lo[i] = make_float4(__fsub_rn(v.x, h.x), __fsub_rn(v.y, h.y), __fsub_rn(v.z, h.z), __fsub_rn(v.w, h.w));
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // generic writes -> tensor core reads
        __syncwarp();
        if (lane == 0) mbar_arrive(conv_bar(s));
      }
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_device_status, kStatusTimeout);
    }
    // stage this CTA's accumulator in shared memory (the ring is free once the MMAs are done)
    bool have = ok && (nk == 0 || mbar_wait(accum_bar, 0u, kWaitNs * 4, abort_flag));
    have = __all_sync(0xffffffffu, have) && !*abort_flag;
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    if (have) {
      tc_fence_after();
      const int r = 32 * q + lane;
      float* row = red + (size_t)r * RED_STRIDE;
      float sr = 1.0f;
      if constexpr (Md::kF16) sr = pow2f(-ea[r]);
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
          for (int i = 0; i < 32; ++i) v[i] = (v[i] * sr) * pow2f(-ew[32 * c + i]);  // exact power-of-two scaling
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
  {
    // Each thread keeps kUnroll float4 positions in flight (remote partials and C loads issued
    // before any is used), so the epilogue streams instead of waiting one load at a time.
    constexpr int kUnroll = 4;
    const int rank = splits > 1 ? (int)cluster_rank() : 0;
    const int rows_per_rank = (BM + splits - 1) / splits;
    const int r0 = rank * rows_per_rank, r1 = (r0 + rows_per_rank < BM) ? r0 + rows_per_rank : BM;
    const bool vec = (N & 3) == 0;
    const uint32_t red_base = smem_u32(red);
    const int total = (r1 - r0) * (BN / 4);
    for (int base = threadIdx.x; base < total; base += THREADS * kUnroll) {
      float4 acc[kUnroll], cc[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int idx = base + u * THREADS;
        acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        cc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (idx >= total) continue;
        const int r = r0 + idx / (BN / 4), c = 4 * (idx % (BN / 4));
        const int64_t m = m0 + r, n = n0 + c;
        if (m >= M || n >= N) continue;
        const uint32_t off = red_base + (uint32_t)((r * RED_STRIDE + c) * 4);
        if (splits > 1) {
          float4 part[MAX_CLUSTER];
#pragma unroll
          for (int qr = 0; qr < MAX_CLUSTER; ++qr)  // all remote loads in flight at once
            if (qr < splits) part[qr] = ld_cluster_f4(map_to_rank(off, (uint32_t)qr));
          acc[u] = part[0];
#pragma unroll
          for (int qr = 1; qr < MAX_CLUSTER; ++qr)  // summed in rank order
            if (qr < splits)
              acc[u] = make_float4(__fadd_rn(acc[u].x, part[qr].x), __fadd_rn(acc[u].y, part[qr].y),
                                   __fadd_rn(acc[u].z, part[qr].z), __fadd_rn(acc[u].w, part[qr].w));
        } else {
          acc[u] = *reinterpret_cast<const float4*>(red + r * RED_STRIDE + c);
        }
        if (C && vec && n + 4 <= N) cc[u] = __ldcs(reinterpret_cast<const float4*>(C + m * N + n));
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int idx = base + u * THREADS;
        if (idx >= total) continue;
        const int r = r0 + idx / (BN / 4), c = 4 * (idx % (BN / 4));
        const int64_t m = m0 + r, n = n0 + c;
        if (m >= M || n >= N) continue;
        float* o = out + m * N + n;
        if (vec && n + 4 <= N) {
          float4 v = acc[u];
          if (C)
            v = make_float4(__fsub_rn(v.x, cc[u].x), __fsub_rn(v.y, cc[u].y), __fsub_rn(v.z, cc[u].z),
                            __fsub_rn(v.w, cc[u].w));
          *reinterpret_cast<float4*>(o) = v;
        } else {
          const float v[4] = {acc[u].x, acc[u].y, acc[u].z, acc[u].w};
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (n + j < N) o[j] = C ? __fsub_rn(v[j], C[m * N + n + j]) : v[j];
        }
      }
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
    tmem_dealloc(tmem, TMEM_COLS);
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

template <class Md>
bool set_smem_attr() {
  static bool done[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (!done[dev]) {
    if (cudaFuncSetAttribute(tc_gemm_kernel<Md>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES) !=
        cudaSuccess)
      return false;
    done[dev] = true;
  }
  return true;
}

// Co-resident clusters of s CTAs (each one SM) on the current device; clusters must fit
// inside one GPC, so this is not simply SMs / s.  Both modes use the same shared memory
// and block shape, so one cache serves both.  Cached per device.
int max_active_clusters(int s, int sms) {
  static int cache[64][MAX_CLUSTER + 1] = {{0}};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return std::max(1, sms / s);
  int& v = cache[dev][s];
  if (v == 0) {
    int n = 0;
    if (set_smem_attr<Tf32x3>()) {
      cudaLaunchConfig_t cfg;
      std::memset(&cfg, 0, sizeof(cfg));
      cfg.gridDim = dim3(1, 1, (unsigned)s);
      cfg.blockDim = dim3(THREADS, 1, 1);
      cfg.dynamicSmemBytes = SMEM_BYTES;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 1;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = (unsigned)s;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      if (cudaOccupancyMaxActiveClusters(&n, tc_gemm_kernel<Tf32x3>, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();
    v = n > 0 ? n : std::max(1, sms / s);
  }
  return v;
}

// Split of the tiles into launches: full waves of unsplit tiles, then the remaining tiles with
// K split across clusters so the last wave is not mostly idle.  Time of a launch ~ waves x
// (kFixedK + K / s), waves counting co-resident clusters of size s; kFixedK is the fixed cost of
// a CTA (launch, pipeline fill, staging and cross-CTA reduction of its 128 KB tile) measured on
// GB300 in units of K.  At least 256 of K per CTA; ties go to fewer splits.
constexpr double kFixedK = 450.0;

int best_split(int64_t tiles, int64_t K, int sms) {
  const int64_t max_s = std::max<int64_t>(1, std::min<int64_t>(MAX_CLUSTER, K / 256));
  int64_t best = 1;
  double best_cost = 1e300;
  for (int64_t s = 1; s <= max_s; ++s) {
    const int64_t clusters = max_active_clusters((int)s, sms);
    const double cost = (double)ceil_div(tiles, clusters) * (kFixedK + (double)K / (double)s);
    if (cost < best_cost * (1.0 - 1e-9)) {
      best_cost = cost;
      best = s;
    }
  }
  return (int)best;
}

struct TcLaunches {
  int64_t full_tiles;  // tiles of the first, unsplit launch (whole waves)
  int64_t rest_tiles;  // tiles of the second launch
  int rest_splits;
};

TcLaunches tc_launches(int64_t M, int64_t K, int64_t N, int sms) {
  const int64_t tiles = ceil_div(M, BM) * ceil_div(N, BN);
  TcLaunches t{0, tiles, 1};
  const int64_t waves = tiles / sms;
  if (waves >= 1) {
    // keep the unsplit waves only if splitting the remainder beats one more unsplit wave
    const int64_t rest = tiles - waves * sms;
    if (rest == 0) return TcLaunches{tiles, 0, 1};
    const int s = best_split(rest, K, sms);
    const double split_cost = (double)ceil_div(rest, max_active_clusters(s, sms)) * (kFixedK + (double)K / s);
    if (split_cost < kFixedK + (double)K) return TcLaunches{waves * sms, rest, s};
    return TcLaunches{0, tiles, 1};
  }
  t.rest_splits = best_split(tiles, K, sms);
  return t;
}

template <class Md>
spl_status launch_tc(const LinearArgs& a, int skip_kblock, int forced_splits) {
  if (!set_smem_attr<Md>()) return SPL_ECUDA;
  TcMaps maps;
  std::memset(&maps, 0, sizeof(maps));
  const int* a_exp = nullptr;
  if constexpr (Md::kF16) {
    // split A (row exponents, hi, lo) into the workspace, then map the two fp16 halves
    char* base = static_cast<char*>(a.ws) + kCounterBytes;
    int* exps = reinterpret_cast<int*>(base);
    uint16_t* a_hi = reinterpret_cast<uint16_t*>(base + round_up(a.M * 4, 256));
    uint16_t* a_lo = reinterpret_cast<uint16_t*>(base + round_up(a.M * 4, 256) + round_up(a.M * a.K * 2, 256));
    const spl_status st = run_split_fp16(a_hi, a_lo, exps, a.a, a.M, a.K, a.stream);
    if (st != SPL_OK) return st;
    a_exp = exps;
    if (!make_map(&maps.a, a_hi, true, a.M, a.K, Md::BK, BM, CU_TENSOR_MAP_SWIZZLE_64B) ||
        !make_map(&maps.a_lo, a_lo, true, a.M, a.K, Md::BK, BM, CU_TENSOR_MAP_SWIZZLE_64B) ||
        !make_map(&maps.w_hi, a.w_h16, true, a.N, a.K, Md::BK, BN, CU_TENSOR_MAP_SWIZZLE_64B) ||
        !make_map(&maps.w_lo, a.w_l16, true, a.N, a.K, Md::BK, BN, CU_TENSOR_MAP_SWIZZLE_64B))
      return SPL_ECUDA;
  } else {
    if (!make_map(&maps.a, a.a, false, a.M, a.K, Md::BK, BM, CU_TENSOR_MAP_SWIZZLE_64B) ||
        !make_map(&maps.w_hi, a.w_hi, false, a.N, a.K, Md::BK, BN, CU_TENSOR_MAP_SWIZZLE_64B) ||
        !make_map(&maps.w_lo, a.w_lo, false, a.N, a.K, Md::BK, BN, CU_TENSOR_MAP_SWIZZLE_64B))
      return SPL_ECUDA;
  }
  const int m_tiles = (int)ceil_div(a.M, BM);
  const TcLaunches t = forced_splits > 0 ? TcLaunches{0, ceil_div(a.M, BM) * ceil_div(a.N, BN), forced_splits}
                                         : tc_launches(a.M, a.K, a.N, device_sm_count());
  auto launch = [&](int64_t tiles, int64_t base, int splits) -> spl_status {
    if (tiles <= 0) return SPL_OK;
    const int64_t kps = round_up(ceil_div(a.K, splits), Md::BK);
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof(cfg));
    cfg.gridDim = dim3((unsigned)tiles, 1, (unsigned)splits);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = a.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = (unsigned)splits;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, tc_gemm_kernel<Md>, maps, a.out, a.c, a_exp,
                                             (const int*)a.w_exp, a.M, a.K, a.N, kps, splits, (int)base, m_tiles,
                                             skip_kblock);
    note_launches(1);
    return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
  };
  spl_status st = launch(t.full_tiles, 0, 1);
  if (st != SPL_OK) return st;
  return launch(t.rest_tiles, t.full_tiles, t.rest_splits);
}

spl_status run_tc_impl(const LinearArgs& a, int skip_kblock, int forced_splits) {
  const int cc = device_cc();
  if (cc != 100 && cc != 103) return SPL_EUNSUPPORTED;
  const bool f16 = a.path == SPL_PATH_FP16X3;
  if (f16) {
    if (!a.w_h16 || !a.w_l16 || !a.w_exp) return SPL_EUNSUPPORTED;
    if ((a.K & 7) != 0) return SPL_EALIGN;  // fp16 rows must be whole 16-byte units
    if (!aligned16(a.w_h16) || !aligned16(a.w_l16)) return SPL_EALIGN;
    if (!a.ws || a.ws_bytes < kCounterBytes + tc_asplit_bytes(a.M, a.K, a.path)) return SPL_EWORKSPACE;
    if (!aligned16(a.ws)) return SPL_EALIGN;
  } else {
    if (!a.w_hi || !a.w_lo) return SPL_EUNSUPPORTED;
    if (!aligned16(a.w_hi) || !aligned16(a.w_lo)) return SPL_EALIGN;
  }
  if (a.M > 0x7fffffffLL || a.N > 0x7fffffffLL || a.K > 0x7fffffffLL) return SPL_ESHAPE;
  if (ceil_div(a.M, BM) * ceil_div(a.N, BN) > 0x7fffffffLL || forced_splits > MAX_CLUSTER) return SPL_ESHAPE;
  return f16 ? launch_tc<Fp16x3>(a, skip_kblock, forced_splits) : launch_tc<Tf32x3>(a, skip_kblock, forced_splits);
}

}  // namespace

size_t tc_asplit_bytes(int64_t M, int64_t K, spl_path path) {
  if (path != SPL_PATH_FP16X3) return 0;
  return (size_t)(round_up(M * 4, 256) + 2 * round_up(M * K * 2, 256));  // exponents, hi, lo
}

Plan plan_tc(int64_t M, int64_t K, int64_t N, int sms, spl_path path) {
  Plan p{};
  p.kernel = kKernelTc;
  const TcLaunches t = tc_launches(M, K, N, sms);
  p.splits = t.rest_splits;
  p.k_per_split = ceil_div(K, t.rest_splits);
  p.ws_asplit = tc_asplit_bytes(M, K, path);  // partials are reduced through distributed shared memory
  return p;
}

spl_status run_tc(const LinearArgs& a, const Plan& p) {
  (void)p;
  return run_tc_impl(a, -1, 0);
}

int tc_uniform_splits(int64_t M, int64_t K, int64_t N) {
  const TcLaunches t = tc_launches(M, K, N, device_sm_count());
  return t.full_tiles > 0 && t.rest_tiles > 0 ? 0 : (t.full_tiles > 0 ? 1 : t.rest_splits);
}

spl_status run_tc_splits(const LinearArgs& a, int splits) {
  if (splits < 1 || splits > MAX_CLUSTER) return SPL_ESHAPE;
  return run_tc_impl(a, -1, splits);
}

}  // namespace spl

// Failure-detection test hook: one TF32X3 product in which the copy of the first K stage is
// never issued, so the kernel's bounded waits run out (about 1 s), it raises the device status
// word and returns.  The paper has no counterpart.
extern "C" spl_status spl_test_tc_wait_timeout(float* out, const float* A, const spl_weight* W, int64_t M, int64_t K,
                                               int64_t N, cudaStream_t stream) {
  using namespace spl;
  if (!out || !A || !W || !W->w || !W->tf32_hi || !W->tf32_lo || M <= 0 || N <= 0 || K <= 0 || (K & 3))
    return SPL_EINVAL;
  if (K > 256) return SPL_ESHAPE;  // one K range per tile: the skipped stage belongs to every CTA
  LinearArgs args{};
  args.out = out;
  args.a = A;
  args.w = W->w;
  args.w_hi = W->tf32_hi;
  args.w_lo = W->tf32_lo;
  args.M = M;
  args.K = K;
  args.N = N;
  args.stream = stream;
  args.path = SPL_PATH_TF32X3;
  return run_tc_impl(args, 0, 0);
}
