// FP32 FMA product on the CUDA cores: out[M, N] = A[M, K] W[N, K]^T (- C).
//
// This is the masked product r = W x~ of Sec. 5.1 (and the correction W eta
// of Sec. 5.2) in plain binary32: every term is one fmaf and each output is
// summed left to right over its K range, so the result obeys the standard
// model the paper's bound is built on (Eq. dot-product-bound, Thm. 4).
//
// Tiling: 128 x 128 output tile per 256-thread block, K step 8, each thread
// owns an 8 x 8 register tile (two 4-row and two 4-column strips 64 apart so
// the shared-memory float4 reads are conflict-free).  Operands are staged in
// shared memory transposed to [k][m] and double-buffered through registers.
// Split-K (blockIdx.z) writes fp32 partials to the workspace; a separate
// kernel sums them in split order and subtracts C (deterministic).

#include <algorithm>

#include "common.cuh"

namespace spl {
namespace {

constexpr int BM = 128, BN = 128, BK = 8, PAD = 4, THREADS = 256;

__global__ void __launch_bounds__(THREADS, 2)
simt_gemm_kernel(float* __restrict__ out, const float* __restrict__ A, const float* __restrict__ W,
                 const float* __restrict__ C, int64_t M, int64_t K, int64_t N, int64_t k_per_split,
                 int splits) {
  __shared__ __align__(16) float As[2][BK][BM + PAD];
  __shared__ __align__(16) float Bs[2][BK][BN + PAD];

  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;
  const int split = blockIdx.z;
  const int64_t kbeg = (int64_t)split * k_per_split;
  const int64_t kend = std::min<int64_t>(K, kbeg + k_per_split);

  // load mapping: one float4 of A and one of W per thread per K step
  const int lrow = tid >> 1, lk = (tid & 1) * 4;
  const int64_t arow = m0 + lrow, wrow = n0 + lrow;
  const float* aptr = A + arow * K;
  const float* wptr = W + wrow * K;

  auto load_a = [&](int64_t k) -> float4 {
    if (arow < M && k + lk < kend) return __ldg(reinterpret_cast<const float4*>(aptr + k + lk));
    return make_float4(0.f, 0.f, 0.f, 0.f);
  };
  auto load_w = [&](int64_t k) -> float4 {
    if (wrow < N && k + lk < kend) return __ldg(reinterpret_cast<const float4*>(wptr + k + lk));
    return make_float4(0.f, 0.f, 0.f, 0.f);
  };
  auto stash = [&](int buf, float4 a, float4 w) {
    As[buf][lk + 0][lrow] = a.x;
    As[buf][lk + 1][lrow] = a.y;
    As[buf][lk + 2][lrow] = a.z;
    As[buf][lk + 3][lrow] = a.w;
    Bs[buf][lk + 0][lrow] = w.x;
    Bs[buf][lk + 1][lrow] = w.y;
    Bs[buf][lk + 2][lrow] = w.z;
    Bs[buf][lk + 3][lrow] = w.w;
  };

  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  int buf = 0;
  if (kbeg < kend) {
    stash(0, load_a(kbeg), load_w(kbeg));
    __syncthreads();
  }
  for (int64_t k = kbeg; k < kend; k += BK) {
    const bool more = k + BK < kend;
    float4 na, nw;
    if (more) {
      na = load_a(k + BK);
      nw = load_w(k + BK);
    }
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      const float4 a0 = *reinterpret_cast<const float4*>(&As[buf][kk][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4*>(&As[buf][kk][64 + ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&Bs[buf][kk][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Bs[buf][kk][64 + tx * 4]);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) {
      stash(buf ^ 1, na, nw);
      __syncthreads();
      buf ^= 1;
    }
  }

  // epilogue
  float* dst = splits > 1 ? out + (int64_t)split * M * N : out;
  const bool vec = (N & 3) == 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t m = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (m >= M) continue;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t n = n0 + h * 64 + tx * 4;
      float v[4] = {acc[i][4 * h + 0], acc[i][4 * h + 1], acc[i][4 * h + 2], acc[i][4 * h + 3]};
      if (splits == 1 && C) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (n + j < N) v[j] = __fsub_rn(v[j], C[m * N + n + j]);
      }
      if (vec && n + 3 < N) {
        *reinterpret_cast<float4*>(dst + m * N + n) = make_float4(v[0], v[1], v[2], v[3]);
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (n + j < N) dst[m * N + n + j] = v[j];
      }
    }
  }
}

__global__ void __launch_bounds__(256) splitk_reduce_kernel(float* __restrict__ out, const float* __restrict__ part,
                                                            const float* __restrict__ C, int splits, int64_t total) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  if ((total & 3) == 0) {
    const int64_t t4 = total >> 2;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < t4; i += stride) {
      float4 s = __ldcg(reinterpret_cast<const float4*>(part) + i);
      for (int sp = 1; sp < splits; ++sp) {
        const float4 p = __ldcg(reinterpret_cast<const float4*>(part + (int64_t)sp * total) + i);
        s = make_float4(__fadd_rn(s.x, p.x), __fadd_rn(s.y, p.y), __fadd_rn(s.z, p.z), __fadd_rn(s.w, p.w));
      }
      if (C) {
        const float4 c = __ldcs(reinterpret_cast<const float4*>(C) + i);
        s = make_float4(__fsub_rn(s.x, c.x), __fsub_rn(s.y, c.y), __fsub_rn(s.z, c.z), __fsub_rn(s.w, c.w));
      }
      reinterpret_cast<float4*>(out)[i] = s;
    }
  } else {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
      float s = __ldcg(part + i);
      for (int sp = 1; sp < splits; ++sp) s = __fadd_rn(s, __ldcg(part + (int64_t)sp * total + i));
      if (C) s = __fsub_rn(s, C[i]);
      out[i] = s;
    }
  }
}

}  // namespace

spl_status run_splitk_reduce(float* out, const float* part, const float* c, int splits, int64_t M, int64_t N,
                             cudaStream_t stream) {
  const int64_t total = M * N;
  if (total == 0) return SPL_OK;
  const int64_t items = (total & 3) == 0 ? total / 4 : total;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(ceil_div(items, 256), (int64_t)device_sm_count() * 8));
  splitk_reduce_kernel<<<grid, 256, 0, stream>>>(out, part, c, splits, total);
  return launch_status();
}

Plan plan_simt(int64_t M, int64_t K, int64_t N, int sms) {
  Plan p{};
  p.kernel = kKernelSimt;
  const int64_t tiles = ceil_div(M, BM) * ceil_div(N, BN);
  const int64_t slots = (int64_t)sms * 2;  // two 256-thread blocks resident per SM
  int64_t s = tiles >= slots ? 1 : std::max<int64_t>(1, slots / std::max<int64_t>(tiles, 1));
  s = std::min<int64_t>(s, std::max<int64_t>(1, K / 256));  // at least 256 K per split
  p.k_per_split = round_up(ceil_div(K, s), BK);
  p.splits = (int)std::max<int64_t>(1, ceil_div(K, p.k_per_split));
  p.ws_partials = p.splits > 1 ? (size_t)round_up((int64_t)p.splits * M * N * 4, 256) : 0;
  return p;
}

spl_status run_simt(const LinearArgs& a, const Plan& p) {
  dim3 grid((unsigned)ceil_div(a.N, BN), (unsigned)ceil_div(a.M, BM), (unsigned)p.splits);
  if (grid.y > 65535u || grid.z > 65535u) return SPL_ESHAPE;
  if (p.splits == 1) {
    simt_gemm_kernel<<<grid, THREADS, 0, a.stream>>>(a.out, a.a, a.w, a.c, a.M, a.K, a.N, p.k_per_split, 1);
    return launch_status();
  }
  float* part = reinterpret_cast<float*>(static_cast<char*>(a.ws) + kCounterBytes);
  simt_gemm_kernel<<<grid, THREADS, 0, a.stream>>>(part, a.a, a.w, nullptr, a.M, a.K, a.N, p.k_per_split,
                                                   p.splits);
  spl_status st = launch_status();
  if (st != SPL_OK) return st;
  return run_splitk_reduce(a.out, part, a.c, p.splits, a.M, a.N, a.stream);
}

}  // namespace spl
