// Streaming decode product for M <= 16 rows: out[M, N] = X~[M, K] W[N, K]^T (- C).
//
// At decode (one new token per step, Sec. 2.2; the paper's server batch is
// 15 prompts, Sec. 6.1) the product reads every weight once and does only M
// FMAs per weight, so it is bound by HBM bandwidth, not by arithmetic.  This
// kernel streams W exactly once with 16-byte cache-streaming loads, keeps the
// K-slice of X~ in shared memory, and fuses the unmask r - W eta (Eq.
// add-and-then-subtract) into the final write.
//
// Work unit: a 256-thread block owns RB consecutive rows of W over one
// K-slice.  Each quarter-warp (8 lanes) reads one row at a time, 32 floats
// (one 128-byte line) per step, so a warp-wide load covers four rows and a
// shared-memory read of X~ is one 128-byte line broadcast to the four
// quarters.  A lane holds RQ rows (rows q, q+4, ... of its warp's 4 RQ) x MT
// partial dot products; at the end each quarter-warp sums its 8 lanes with a
// reduce-scatter butterfly (V - 1 shuffles for V = RQ MT values, not 3 V).
// Every output element is summed in one order whatever MT and RQ are: the
// lane's own k positions in increasing order, then the fixed xor-4/2/1 tree
// over the 8 lanes, then the K-slices in split order; so a correction
// computed with a different number of rows per launch cancels exactly.
//
// The K-split is a multiple of 128 elements and is sized so the grid fills the
// SMs.  With more than one split, each block writes fp32 partials to the
// workspace and bumps an arrival counter; the last block of a row group sums
// the partials in split order (deterministic), subtracts C, writes the result
// and resets the counter to zero.

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "noise.cuh"

namespace spl {
namespace {

constexpr int THREADS = 256, WARPS = 8;
constexpr int kStep = 32;                    // K elements a quarter-warp covers per step
constexpr int kSliceAlign = 64;              // K-slices are multiples of this (staged_ks pads the
                                             // staged slice to the iteration step)
constexpr int kXsBytes = 96 * 1024;          // largest X~ slice a block stages (two blocks per SM)
constexpr int kMaxKs = kXsBytes / (4 * kGemvMaxM) / kSliceAlign * kSliceAlign;  // 1536: every MT fits it

// Rows per lane: 4 while the accumulators are few (MT <= 2), else 2 (RQ x MT accumulators).
__host__ __device__ constexpr int rows_per_lane(int mt) { return mt <= 2 ? 4 : 2; }
__host__ __device__ constexpr int rows_per_block(int mt) { return WARPS * 4 * rows_per_lane(mt); }
// Steps of 32 per unrolled iteration: 8 float4 loads of W in flight per lane per buffer, but 4 at 8
// rows (then 80 registers give 3 blocks per SM instead of 2; measured faster at 8 rows, slower at 16).
__host__ __device__ constexpr int unroll_steps(int mt) { return mt == 8 ? 2 : 8 / rows_per_lane(mt); }
// Columns of the staged X~ slice: ks rounded up to the columns one unrolled iteration reads (64 or
// 128), so a slice that is a multiple of kSliceAlign but not of that step is staged with zero
// columns after it and no iteration reads past the staged rows.
__host__ __device__ constexpr int staged_ks(int mt, int ks) {
  return (ks + unroll_steps(mt) * kStep - 1) / (unroll_steps(mt) * kStep) * (unroll_steps(mt) * kStep);
}

// Rows of X~ are summed in packed pairs (p2 / fma2 / up2 of noise.cuh): one fma.rn.f32x2 does the
// two round-to-nearest FMAs the scalar loop would, so the sums are the same bit for bit with half
// the FMA instructions.
__device__ __forceinline__ void lds_v2b64(uint32_t addr, unsigned long long& a, unsigned long long& b) {
  asm volatile("ld.shared.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "r"(addr));
}

// Paired layout of the staged X~ (MT >= 4): rows 2p and 2p + 1 interleaved, and within each step of
// 32 columns the 16-byte group that lane i reads first holds columns 4i, 4i + 1 of both rows and
// the second one columns 4i + 2, 4i + 3: a quarter-warp reads 128 contiguous bytes per access.
// Offset (in floats) of the group holding columns k, k + 1 (k = 4q + 2h) of pair p.
__device__ __forceinline__ int pair_off(int p, int ks, int q, int h) {
  return p * 2 * ks + (q >> 3) * 64 + h * 32 + (q & 7) * 4;
}

// Reduce-scatter over the 8 lanes of a quarter-warp (xor offsets 4, 2, 1).  While C >= 2 values
// remain, the lane with bit O set keeps the upper half and sends the lower half; afterwards the
// single value left is summed with a plain xor exchange.  Each step adds (own, partner), so every
// element gets the same tree whatever C is.
template <int C, int O, int V>
__device__ __forceinline__ void quarter_reduce(float (&v)[V], int lane) {
  if constexpr (O >= 1) {
    if constexpr (C >= 2) {
      const bool up = (lane & O) != 0;
#pragma unroll
      for (int i = 0; i < C / 2; ++i) {
        const float send = up ? v[i] : v[i + C / 2];
        const float keep = up ? v[i + C / 2] : v[i];
        v[i] = __fadd_rn(keep, __shfl_xor_sync(0xffffffffu, send, O));
      }
      quarter_reduce<C / 2, O / 2, V>(v, lane);
    } else {
      v[0] = __fadd_rn(v[0], __shfl_xor_sync(0xffffffffu, v[0], O));
      quarter_reduce<1, O / 2, V>(v, lane);
    }
  }
}

// Index (in the lane's original V values) of the first value the lane holds after quarter_reduce,
// and the mask of lane bits whose partners hold the same values.
template <int V>
__device__ __forceinline__ int reduced_base(int lane, int* dup_mask) {
  int base = 0, c = V, dup = 0;
#pragma unroll
  for (int o = 4; o >= 1; o >>= 1) {
    if (c >= 2) {
      if (lane & o) base += c / 2;
      c /= 2;
    } else {
      dup |= o;
    }
  }
  *dup_mask = dup;
  return base;
}

constexpr int kNoMask = -1;

// Noise of the fused mask, as the kernel receives it (MASK != kNoMask).
struct KernelNoise {
  float* xt;
  float b;
  PhiloxKey key;
  uint64_t offset;
  const uint64_t* offset_dev;
  int x_rows;        // rows from x_rows on: noise alone, drawn delta blocks further on, counters from row x_rows
  uint64_t delta;
};

template <int MT, int MASK>
__global__ void __launch_bounds__(THREADS)
gemv_kernel(float* __restrict__ out, const float* __restrict__ X, const float* __restrict__ W,
            const float* __restrict__ C, float* __restrict__ part, unsigned int* __restrict__ counters, int M,
            int64_t K, int64_t N, int ks, int splits, int prefetch_lines, const __grid_constant__ KernelNoise nz,
            int c_rows) {
  constexpr int RQ = rows_per_lane(MT), RB = rows_per_block(MT), U = unroll_steps(MT);
  constexpr int V = RQ * MT;
  extern __shared__ __align__(16) float4 xs[];  // [MT][staged_ks(MT, ks) / 4]
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = lane >> 3, kl = (lane & 7) * 4;
  const int split = blockIdx.y;
  const int64_t k0 = (int64_t)split * ks;
  const int klen = (int)(K - k0 < ks ? K - k0 : (int64_t)ks);  // multiple of 4
  const int64_t row0 = (int64_t)blockIdx.x * RB + warp * 4 * RQ + quarter;  // lane's rows: row0 + 4 r

  const float* wp[RQ];
  bool valid[RQ];
#pragma unroll
  for (int r = 0; r < RQ; ++r) {
    valid[r] = row0 + 4 * r < N;
    wp[r] = W + (valid[r] ? row0 + 4 * r : 0) * K + k0 + kl;
  }

  // W never changes, so its first lines are fetched before waiting on the kernel that writes X~
  // and C: the first U steps into registers (after the staging when it draws noise, which needs
  // the registers), the next prefetch_lines lines of each row into L2.
  float4 w[U][RQ];
  auto load_first = [&]() {
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int r = 0; r < RQ; ++r)
        w[u][r] = (valid[r] && u * kStep + kl < klen) ? __ldcs(reinterpret_cast<const float4*>(wp[r] + u * kStep))
                                                       : make_float4(0.f, 0.f, 0.f, 0.f);
  };
  if constexpr (MASK == kNoMask) load_first();
  for (int l = (MASK == kNoMask ? U : 0) + (lane & 7); l < prefetch_lines && l * kStep < klen; l += 8)
#pragma unroll
    for (int r = 0; r < RQ; ++r)
      if (valid[r]) asm volatile("prefetch.global.L2 [%0];" ::"l"(wp[r] - kl + l * kStep));
  pdl_wait();
  // the next kernel may be scheduled now: its blocks take the slots this grid leaves free and
  // fetch their first weight lines while this one streams (decode 2.28 -> 2.24 ms per token)
  pdl_trigger();

  // stage X~[:, k0:k0+ks] (rows >= M and columns >= klen are zero), rows ksp columns apart
  const int ksp = staged_ks(MT, ks);
  const int q_row = ksp >> 2, q_len = klen >> 2;
  float* xsf = reinterpret_cast<float*>(xs);
  // X~ of rows m, columns 4q..4q+3 (stored as given, or with the noise drawn here)
  auto x4 = [&](int m, int q, float4* dst_out) -> float4 {
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (m < M && q < q_len) {
      const bool own = MASK == kNoMask || m < nz.x_rows;  // a row of X (else noise alone)
      if (own) v = __ldg(reinterpret_cast<const float4*>(X + (int64_t)m * K + k0) + q);
      if constexpr (MASK != kNoMask) {
        const int64_t mr = own ? m : m - nz.x_rows;
        const uint64_t j = (uint64_t)((mr * K + k0) >> 2) + (uint64_t)q + nz.offset + (own ? 0ull : nz.delta) +
                           (nz.offset_dev ? *nz.offset_dev : 0ull);
        v = add4(v, draw_block<MASK>(j, nz.key, nz.b));
        if (dst_out) __stcs(dst_out, v);
      }
    }
    return v;
  };
  if constexpr (MT >= 4) {
    // fused mask: X~ = fl32(X + eta), eta of element (m, k) being lane k % 4 of Philox block
    // (m K + k) / 4 + offset, as the mask kernel draws it; the first row group writes X~ out
    const bool write_xt = MASK != kNoMask && blockIdx.x == 0;
#pragma unroll
    for (int p = 0; p < MT / 2; ++p)
      for (int q = threadIdx.x; q < q_row; q += THREADS) {
        float4* d0 = write_xt && 2 * p < M && q < q_len ? reinterpret_cast<float4*>(nz.xt + (int64_t)(2 * p) * K + k0) + q : nullptr;
        float4* d1 = write_xt && 2 * p + 1 < M && q < q_len ? reinterpret_cast<float4*>(nz.xt + (int64_t)(2 * p + 1) * K + k0) + q : nullptr;
        const float4 a = x4(2 * p, q, d0), b = x4(2 * p + 1, q, d1);
        *reinterpret_cast<float4*>(xsf + pair_off(p, ksp, q, 0)) = make_float4(a.x, b.x, a.y, b.y);
        *reinterpret_cast<float4*>(xsf + pair_off(p, ksp, q, 1)) = make_float4(a.z, b.z, a.w, b.w);
      }
    if constexpr (MASK != kNoMask) load_first();
  } else if constexpr (MASK == kNoMask) {
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      const float4* src = reinterpret_cast<const float4*>(X + (int64_t)m * K + k0);
      for (int q = threadIdx.x; q < q_row; q += THREADS)
        xs[m * q_row + q] = (m < M && q < q_len) ? __ldg(src + q) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  } else {
    // fused mask: X~ = fl32(X + eta), eta of element (m, k) being lane k % 4 of Philox block
    // (m K + k) / 4 + offset, as the mask kernel draws it; the blocks of the first row group
    // also write X~ out
    const uint64_t off = nz.offset + (nz.offset_dev ? *nz.offset_dev : 0ull);
    const bool write_xt = blockIdx.x == 0;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      const bool own = m < nz.x_rows;  // a row of X (else noise alone, delta blocks further on)
      const float4* src = reinterpret_cast<const float4*>(X + (int64_t)(own ? m : 0) * K + k0);
      float4* dst = reinterpret_cast<float4*>(nz.xt + (int64_t)m * K + k0);
      const int64_t mr = own ? m : m - nz.x_rows;
      const uint64_t j0 = (uint64_t)((mr * K + k0) >> 2) + off + (own ? 0ull : nz.delta);
      for (int q = threadIdx.x; q < q_row; q += THREADS) {
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (m < M && q < q_len) {
          const float4 e = draw_block<MASK>(j0 + (uint64_t)q, nz.key, nz.b);
          v = own ? add4(__ldg(src + q), e) : e;
          if (write_xt) __stcs(dst + q, v);
        }
        xs[m * q_row + q] = v;
      }
    }
    load_first();
  }
  __syncthreads();

  float acc[V];
#pragma unroll
  for (int i = 0; i < V; ++i) acc[i] = 0.f;

  if constexpr (MT >= 4) {
    // acc2[r][p]: rows 2p, 2p + 1 of X~ against the lane's row r of W, as packed pairs
    unsigned long long acc2[RQ][MT / 2];
#pragma unroll
    for (int r = 0; r < RQ; ++r)
#pragma unroll
      for (int p = 0; p < MT / 2; ++p) acc2[r][p] = 0ull;
    const uint32_t xbase = static_cast<uint32_t>(__cvta_generic_to_shared(xsf));
    for (int kb = 0; kb < klen; kb += U * kStep) {
      float4 wn[U][RQ];
      const int kn = kb + U * kStep;
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int r = 0; r < RQ; ++r)
          wn[u][r] = (valid[r] && kn + u * kStep + kl < klen)
                         ? __ldcs(reinterpret_cast<const float4*>(wp[r] + kn + u * kStep))
                         : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        unsigned long long wx[RQ], wy[RQ], wz[RQ], ww[RQ];
#pragma unroll
        for (int r = 0; r < RQ; ++r) {
          wx[r] = p2(w[u][r].x, w[u][r].x);
          wy[r] = p2(w[u][r].y, w[u][r].y);
          wz[r] = p2(w[u][r].z, w[u][r].z);
          ww[r] = p2(w[u][r].w, w[u][r].w);
        }
        const int q = (kb + u * kStep + kl) >> 2;
#pragma unroll
        for (int p = 0; p < MT / 2; ++p) {
          unsigned long long x0, x1, x2, x3;  // columns k, k+1, k+2, k+3 of rows 2p, 2p+1
          lds_v2b64(xbase + 4u * (uint32_t)pair_off(p, ksp, q, 0), x0, x1);
          lds_v2b64(xbase + 4u * (uint32_t)pair_off(p, ksp, q, 1), x2, x3);
#pragma unroll
          for (int r = 0; r < RQ; ++r) {
            unsigned long long a = acc2[r][p];
            a = fma2(wx[r], x0, a);
            a = fma2(wy[r], x1, a);
            a = fma2(wz[r], x2, a);
            a = fma2(ww[r], x3, a);
            acc2[r][p] = a;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int r = 0; r < RQ; ++r) w[u][r] = wn[u][r];
    }
#pragma unroll
    for (int r = 0; r < RQ; ++r)
#pragma unroll
      for (int p = 0; p < MT / 2; ++p) up2(acc2[r][p], acc[r * MT + 2 * p], acc[r * MT + 2 * p + 1]);
  }

  const float4* xl = xs + (kl >> 2);
  for (int kb = 0; kb < (MT >= 4 ? 0 : klen); kb += U * kStep) {
    // the next U steps of W while this one is summed
    float4 wn[U][RQ];
    const int kn = kb + U * kStep;
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int r = 0; r < RQ; ++r)
        wn[u][r] = (valid[r] && kn + u * kStep + kl < klen)
                       ? __ldcs(reinterpret_cast<const float4*>(wp[r] + kn + u * kStep))
                       : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        const float4 x = xl[m * q_row + ((kb + u * kStep) >> 2)];
#pragma unroll
        for (int r = 0; r < RQ; ++r) {
          float a = acc[r * MT + m];
          a = fmaf(w[u][r].x, x.x, a);
          a = fmaf(w[u][r].y, x.y, a);
          a = fmaf(w[u][r].z, x.z, a);
          a = fmaf(w[u][r].w, x.w, a);
          acc[r * MT + m] = a;
        }
      }
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int r = 0; r < RQ; ++r) w[u][r] = wn[u][r];
  }

  quarter_reduce<V, 4, V>(acc, lane);
  int dup = 0;
  const int base = reduced_base<V>(lane, &dup);
  constexpr int HELD = V >= 8 ? V / 8 : 1;
  const bool writer = (lane & dup) == 0;

  if (splits == 1) {
    if (writer) {
#pragma unroll
      for (int i = 0; i < HELD; ++i) {
        const int idx = base + i, r = idx / MT, m = idx - r * MT;
        const int64_t n = row0 + 4 * r;
        if (m < M && n < N) {
          const int64_t o = (int64_t)m * N + n;
          out[o] = (C && m < c_rows) ? __fsub_rn(acc[i], C[o]) : acc[i];
        }
      }
    }
    return;
  }

  float* mypart = part + (int64_t)split * M * N;
  if (writer) {
#pragma unroll
    for (int i = 0; i < HELD; ++i) {
      const int idx = base + i, r = idx / MT, m = idx - r * MT;
      const int64_t n = row0 + 4 * r;
      if (m < M && n < N) __stcg(mypart + (int64_t)m * N + n, acc[i]);
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const unsigned int prev = atomicAdd(counters + blockIdx.x, 1u);
    s_last = (prev == (unsigned int)(splits - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int64_t n0 = (int64_t)blockIdx.x * RB;
  for (int idx = threadIdx.x; idx < RB * M; idx += THREADS) {
    const int m = idx / RB;
    const int64_t n = n0 + (idx - m * RB);
    if (n >= N) continue;
    const int64_t o = (int64_t)m * N + n;
    float s = __ldcg(part + o);
    for (int sp = 1; sp < splits; ++sp) s = __fadd_rn(s, __ldcg(part + (int64_t)sp * M * N + o));
    out[o] = (C && m < c_rows) ? __fsub_rn(s, C[o]) : s;
  }
  if (threadIdx.x == 0) counters[blockIdx.x] = 0u;
}

int padded_m(int64_t M) { return M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : M <= 8 ? 8 : 16; }

template <int MT, int MASK = kNoMask>
void* kernel_ptr() { return reinterpret_cast<void*>(gemv_kernel<MT, MASK>); }

void* kernel_for(int mt) {
  switch (mt) {
    case 1: return kernel_ptr<1>();
    case 2: return kernel_ptr<2>();
    case 4: return kernel_ptr<4>();
    case 8: return kernel_ptr<8>();
    default: return kernel_ptr<16>();
  }
}

// Opt every instantiation into the shared memory of the largest X~ slice (once per device).
bool smem_attr_set() {
  static std::mutex mu;
  static bool done[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    void* const kernels[] = {kernel_ptr<1>(), kernel_ptr<2>(), kernel_ptr<4>(), kernel_ptr<8>(), kernel_ptr<16>(),
                             kernel_ptr<1, kZero>(), kernel_ptr<2, kZero>(), kernel_ptr<4, kZero>(),
                             kernel_ptr<1, kLaplace>(), kernel_ptr<2, kLaplace>(), kernel_ptr<4, kLaplace>(),
                             kernel_ptr<1, kGaussian>(), kernel_ptr<2, kGaussian>(), kernel_ptr<4, kGaussian>()};
    for (void* k : kernels)
      if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kXsBytes) != cudaSuccess) {
        cudaGetLastError();
        return false;
      }
    done[dev] = true;
  }
  return true;
}

template <int MT, int MASK = kNoMask>
spl_status launch(const LinearArgs& a, const Plan& p, float* part, unsigned int* counters,
                  const KernelNoise& nz = KernelNoise{}) {
  if (!smem_attr_set()) return SPL_ECUDA;
  dim3 grid((unsigned)ceil_div(a.N, rows_per_block(MT)), (unsigned)p.splits);
  const size_t smem = (size_t)MT * staged_ks(MT, (int)p.k_per_split) * sizeof(float);
  // L2 budget of the early prefetch: about 32 MB over the whole grid, in 128-byte lines per row
  const int64_t rows = (int64_t)grid.x * rows_per_block(MT) * p.splits;
  const int lines = (int)std::min<int64_t>(p.k_per_split / kStep, ((int64_t(32) << 20) / std::max<int64_t>(rows, 1)) >> 7);
  return launch_pdl(gemv_kernel<MT, MASK>, grid, dim3(THREADS), smem, a.stream, a.out, a.a, a.w, a.c, part, counters,
                    (int)a.M, a.K, a.N, (int)p.k_per_split, p.splits, lines, nz, (int)a.c_rows);
}

template <int MASK>
spl_status launch_masked(const LinearArgs& a, const Plan& p, float* part, unsigned int* counters,
                         const KernelNoise& nz) {
  switch (padded_m(a.M)) {
    case 1: return launch<1, MASK>(a, p, part, counters, nz);
    case 2: return launch<2, MASK>(a, p, part, counters, nz);
    default: return launch<4, MASK>(a, p, part, counters, nz);
  }
}

// Resident blocks per SM of the decode kernel for MT rows and a K-slice of ks (cached).
int blocks_per_sm(int mt, int64_t ks) {
  static std::mutex mu;
  static int cache[64][5][kMaxKs / kSliceAlign + 1] = {{{0}}};  // device, log2(mt), ks / kSliceAlign
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (!smem_attr_set()) return 1;
  const int mi = mt == 1 ? 0 : mt == 2 ? 1 : mt == 4 ? 2 : mt == 8 ? 3 : 4;
  const int ki = (int)std::min<int64_t>(kMaxKs / kSliceAlign, ks / kSliceAlign);
  std::lock_guard<std::mutex> lock(mu);
  int& v = cache[dev][mi][ki];
  if (v == 0) {
    int n = 0;
    const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel_for(mt), THREADS,
                                                                         (size_t)mt * staged_ks(mt, (int)ks) * sizeof(float));
    if (e != cudaSuccess) cudaGetLastError();
    v = (e == cudaSuccess && n > 0) ? n : 1;
  }
  return v;
}

}  // namespace

int64_t gemv_max_ks(int64_t M) {
  return std::min<int64_t>(kMaxKs, (int64_t)kXsBytes / (4 * padded_m(M)) / kSliceAlign * kSliceAlign);
}

// K-split of the decode kernel: the number of splits s minimises waves(s) x (K/s + F), waves
// counting the resident block slots of all SMs, with K/s a multiple of 64 no larger than 1536
// (the slice 16 rows can stage, so a correction of up to 16 rows per launch reproduces the
// online order); F (the fixed cost of a block -- staging X~, the warp reduction, the split-K
// reduction -- in units of K) measured on GB300.
constexpr double kGemvFixedK = 512.0;

Plan plan_gemv(int64_t M, int64_t K, int64_t N, int sms) {
  Plan p{};
  p.kernel = kKernelGemv;
  const int mt = padded_m(M);
  const int64_t ks_max = kMaxKs;
  const int64_t groups = ceil_div(N, rows_per_block(mt));
  const int64_t s_min = ceil_div(K, ks_max);
  const int64_t s_max = std::max<int64_t>(s_min, std::min<int64_t>(64, K / 128));
  double best = 1e300;
  for (int64_t s = s_min; s <= s_max; ++s) {
    const int64_t ks = std::min<int64_t>(round_up(ceil_div(K, s), kSliceAlign), ks_max);
    const int64_t splits = ceil_div(K, ks);
    const int64_t slots = (int64_t)sms * blocks_per_sm(mt, ks);
    const double cost = (double)ceil_div(groups * splits, slots) * ((double)ks + kGemvFixedK);
    if (cost < best * (1.0 - 1e-9)) {
      best = cost;
      p.k_per_split = ks;
      p.splits = (int)splits;
    }
  }
  if (p.splits > 1) p.ws_partials = (size_t)round_up((int64_t)p.splits * M * N * 4, 256);
  return p;
}

namespace {
spl_status scratch(const LinearArgs& a, const Plan& p, float** part, unsigned int** counters) {
  *part = nullptr;
  *counters = nullptr;
  if (p.splits > 65535) return SPL_ESHAPE;
  if (p.splits > 1) {
    if (ceil_div(a.N, rows_per_block(padded_m(a.M))) > kMaxCounters) return SPL_ESHAPE;
    *counters = static_cast<unsigned int*>(a.ws);
    *part = reinterpret_cast<float*>(static_cast<char*>(a.ws) + kCounterBytes);
  }
  return SPL_OK;
}
}  // namespace

spl_status run_gemv_masked(const LinearArgs& a, const Plan& p, const MaskNoise& nz) {
  if (a.M > kGemvMaskMaxM || !nz.xt) return SPL_EINVAL;
  float* part;
  unsigned int* counters;
  spl_status st = scratch(a, p, &part, &counters);
  if (st != SPL_OK) return st;
  KernelNoise kn{};
  kn.xt = nz.xt;
  kn.b = nz.b;
  kn.key = make_philox_key(nz.seed, nz.stream_id);
  kn.offset = nz.offset;
  kn.offset_dev = nz.offset_dev;
  kn.x_rows = nz.x_rows < 0 ? (int)a.M : (int)nz.x_rows;
  kn.delta = nz.noise_delta;
  if (nz.b == 0.0f) return launch_masked<kZero>(a, p, part, counters, kn);
  if (nz.mech == SPL_MECH_LAPLACE) return launch_masked<kLaplace>(a, p, part, counters, kn);
  return launch_masked<kGaussian>(a, p, part, counters, kn);
}

spl_status run_gemv(const LinearArgs& a, const Plan& p) {
  float* part;
  unsigned int* counters;
  spl_status st = scratch(a, p, &part, &counters);
  if (st != SPL_OK) return st;
  switch (padded_m(a.M)) {
    case 1: return launch<1>(a, p, part, counters);
    case 2: return launch<2>(a, p, part, counters);
    case 4: return launch<4>(a, p, part, counters);
    case 8: return launch<8>(a, p, part, counters);
    default: return launch<16>(a, p, part, counters);
  }
}

}  // namespace spl

// ---- variant without allocation ---------------------------------------------
// Some callers cannot call cudaMalloc when they need this product: a decode
// loop that must not stall (cudaMalloc and cudaFree synchronise the device),
// a process whose device memory is already fully reserved by another
// allocator, or a worker whose memory budget is fixed when it starts.  For
// them the decode kernel's scratch (arrival counters + split-K partials, the
// same layout as a workspace) lives in this fixed array instead.  Every GPU
// that loads the library holds it until the process exits.
namespace spl {
namespace {

constexpr size_t kStaticPartialBytes = size_t(4) << 20;  // 4 MiB of split-K partials
constexpr size_t kStaticScratchBytes = kCounterBytes + kStaticPartialBytes;
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDev = 64;
std::mutex g_static_mu;
void* g_static_ptr[kMaxDev] = {nullptr};

// Device address of g_static_scratch on the current device, looked up on every call
// (cudaGetSymbolAddress allocates nothing), so that an address from before a cudaDeviceReset is
// never reused.  When the address is new for this device (its first call, or the module was
// loaded again) a clear of the counter region is queued on the caller's stream, ahead of the
// kernel that uses it; the array is zero when the module loads and every call that completes
// leaves the counters at zero, so the clear is only a safeguard.
spl_status static_scratch(void** out, cudaStream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return SPL_ECUDA;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return SPL_ECUDA;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (g_static_ptr[dev] != p) {
    if (cudaMemsetAsync(p, 0, kCounterBytes, stream) != cudaSuccess) return SPL_ECUDA;
    g_static_ptr[dev] = p;
  }
  *out = p;
  return SPL_OK;
}

}  // namespace
}  // namespace spl

extern "C" spl_status spl_masked_linear_unmask_noalloc(float* Y, const float* Xt, const float* W, const float* C,
                                                       int64_t M, int64_t K, int64_t N, cudaStream_t stream) {
  using namespace spl;
  if (M < 0 || K < 0 || N < 0) return SPL_EINVAL;
  if (M == 0 || N == 0) return SPL_OK;
  if (M > kGemvMaxM) return SPL_ESHAPE;
  if (!Y || !C || (K > 0 && (!Xt || !W))) return SPL_EINVAL;
  if ((K & 3) != 0) return SPL_EALIGN;
  if (!aligned16(Y) || !aligned16(C) || (Xt && !aligned16(Xt)) || (W && !aligned16(W))) return SPL_EALIGN;
  if (K > (int64_t(1) << 31) || N > (int64_t(1) << 31)) return SPL_ESHAPE;
  if (K == 0) {
    if (cudaMemsetAsync(Y, 0, (size_t)(M * N) * sizeof(float), stream) != cudaSuccess) return SPL_ECUDA;
    return spl_unmask(Y, Y, C, M, N, stream);
  }
  const Plan plan = plan_gemv(M, K, N, device_sm_count());
  if (plan.ws_partials > kStaticPartialBytes) return SPL_EWORKSPACE;  // beyond the built-in 4 MiB
  if (plan.splits > 1 && ceil_div(N, rows_per_block(padded_m(M))) > kMaxCounters) return SPL_EWORKSPACE;
  void* ws = nullptr;
  spl_status st = static_scratch(&ws, stream);
  if (st != SPL_OK) return st;
  LinearArgs args{};
  args.out = Y;
  args.a = Xt;
  args.w = W;
  args.c = C;
  args.M = M;
  args.K = K;
  args.N = N;
  args.ws = ws;
  args.ws_bytes = kStaticScratchBytes;
  args.stream = stream;
  args.c_rows = M;
  args.path = SPL_PATH_FP32;
  return run_gemv(args, plan);
}
