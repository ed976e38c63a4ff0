// Streaming decode product for M <= 16 rows: out[M, N] = X~[M, K] W[N, K]^T (- C).
//
// At decode (one new token per step, Sec. 2.2; the paper's server batch is
// 15 prompts, Sec. 6.1) the product reads every weight once and does only M
// FMAs per weight, so it is bound by HBM bandwidth, not by arithmetic.  This
// kernel streams W exactly once with 16-byte cache-streaming loads, keeps the
// K-slice of X~ in shared memory, and fuses the unmask r - W eta (Eq.
// add-and-then-subtract) into the final write.
//
// Work unit: a 256-thread block owns 32 (M <= 4) or 16 consecutive rows of W
// over one K-slice; lanes stride the slice in float4 steps and every lane
// keeps 4 x M partial dot products in registers, reduced across the warp
// with shuffles at the end.  The K-split is a multiple of 128 elements and
// is sized so the grid fills the SMs.  With more than one split, each block
// writes fp32 partials to the workspace and bumps an arrival counter; the
// last block of a row group sums the partials in split order (deterministic),
// subtracts C, writes the result and resets the counter to zero.

#include <algorithm>
#include <mutex>

#include "common.cuh"

namespace spl {
namespace {

constexpr int THREADS = 256, WARPS = 8;
constexpr int SMEM_FLOATS = 12000;  // just under 48 KB of X~ slice (static smem adds a few bytes)

// Rows of W per warp: 4 for M <= 4, 2 for larger M (bounds the rows x M accumulators and keeps
// four blocks resident per SM).
constexpr int rows_per_warp(int mt) { return mt >= 8 ? 2 : 4; }

template <int MT, int ROWS_PER_WARP>
__global__ void __launch_bounds__(THREADS)
gemv_kernel(float* __restrict__ out, const float* __restrict__ X, const float* __restrict__ W,
            const float* __restrict__ C, float* __restrict__ part, unsigned int* __restrict__ counters, int M,
            int64_t K, int64_t N, int64_t ks, int splits, int64_t prefetch_bytes) {
  constexpr int ROWS_PER_BLOCK = WARPS * ROWS_PER_WARP;
  extern __shared__ __align__(16) float xs[];  // [MT][ks]
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.y;
  const int64_t k0 = (int64_t)split * ks;
  const int64_t klen = std::min<int64_t>(ks, K - k0);  // multiple of 4

  // the first prefetch_bytes of each of this warp's W rows (slice k0..k0+klen) into L2
  {
    const int64_t n_first = (int64_t)blockIdx.x * ROWS_PER_BLOCK + warp * ROWS_PER_WARP;
    const int64_t lines = std::min<int64_t>(prefetch_bytes, klen * 4) >> 7;  // 128-byte lines per row
    for (int r = 0; r < ROWS_PER_WARP; ++r) {
      if (n_first + r >= N) break;
      const char* base = reinterpret_cast<const char*>(W + (n_first + r) * K + k0);
      for (int64_t l = lane; l < lines; l += 32) asm volatile("prefetch.global.L2 [%0];" ::"l"(base + 128 * l));
    }
  }
  pdl_wait();

  // stage X~[:, k0:k0+klen] (rows >= M are zero)
  const int64_t q_per_row = klen >> 2;
  for (int64_t q = threadIdx.x; q < (int64_t)MT * q_per_row; q += THREADS) {
    const int m = (int)(q / q_per_row);
    const int64_t kq = (q - (int64_t)m * q_per_row) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (m < M) v = __ldg(reinterpret_cast<const float4*>(X + (int64_t)m * K + k0 + kq));
    *reinterpret_cast<float4*>(xs + (int64_t)m * ks + kq) = v;
  }
  __syncthreads();

  const int64_t nbase = (int64_t)blockIdx.x * ROWS_PER_BLOCK + warp * ROWS_PER_WARP;
  const float* wrow[ROWS_PER_WARP];
  bool valid[ROWS_PER_WARP];
#pragma unroll
  for (int r = 0; r < ROWS_PER_WARP; ++r) {
    valid[r] = nbase + r < N;
    wrow[r] = W + (valid[r] ? (nbase + r) : 0) * K + k0;
  }

  float acc[ROWS_PER_WARP][MT];
#pragma unroll
  for (int r = 0; r < ROWS_PER_WARP; ++r)
#pragma unroll
    for (int m = 0; m < MT; ++m) acc[r][m] = 0.f;

#pragma unroll 2
  for (int64_t kk = lane * 4; kk < klen; kk += 128) {
    float4 wv[ROWS_PER_WARP];
#pragma unroll
    for (int r = 0; r < ROWS_PER_WARP; ++r)
      wv[r] = valid[r] ? __ldcs(reinterpret_cast<const float4*>(wrow[r] + kk)) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      const float4 xv = *reinterpret_cast<const float4*>(xs + (int64_t)m * ks + kk);
#pragma unroll
      for (int r = 0; r < ROWS_PER_WARP; ++r) {
        float a = acc[r][m];
        a = fmaf(wv[r].x, xv.x, a);
        a = fmaf(wv[r].y, xv.y, a);
        a = fmaf(wv[r].z, xv.z, a);
        a = fmaf(wv[r].w, xv.w, a);
        acc[r][m] = a;
      }
    }
  }

  pdl_trigger();  // W is streamed: the next kernel may be scheduled

  // warp reduction: lane 0 ends with the full sums
#pragma unroll
  for (int r = 0; r < ROWS_PER_WARP; ++r)
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      float v = acc[r][m];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
      acc[r][m] = v;
    }

  if (splits == 1) {
    if (lane == 0) {
#pragma unroll
      for (int r = 0; r < ROWS_PER_WARP; ++r) {
        if (!valid[r]) continue;
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          if (m >= M) break;
          const int64_t o = (int64_t)m * N + nbase + r;
          out[o] = C ? __fsub_rn(acc[r][m], C[o]) : acc[r][m];
        }
      }
    }
    return;
  }

  float* mypart = part + (int64_t)split * M * N;
  if (lane == 0) {
#pragma unroll
    for (int r = 0; r < ROWS_PER_WARP; ++r) {
      if (!valid[r]) continue;
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        if (m >= M) break;
        __stcg(mypart + (int64_t)m * N + nbase + r, acc[r][m]);
      }
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
  const int64_t n0 = (int64_t)blockIdx.x * ROWS_PER_BLOCK;
  for (int idx = threadIdx.x; idx < ROWS_PER_BLOCK * M; idx += THREADS) {
    const int m = idx / ROWS_PER_BLOCK;
    const int64_t n = n0 + (idx % ROWS_PER_BLOCK);
    if (n >= N) continue;
    const int64_t o = (int64_t)m * N + n;
    float s = __ldcg(part + o);
    for (int sp = 1; sp < splits; ++sp) s = __fadd_rn(s, __ldcg(part + (int64_t)sp * M * N + o));
    out[o] = C ? __fsub_rn(s, C[o]) : s;
  }
  if (threadIdx.x == 0) counters[blockIdx.x] = 0u;
}

int padded_m(int64_t M) { return M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : M <= 8 ? 8 : 16; }

template <int MT>
spl_status launch(const LinearArgs& a, const Plan& p, float* part, unsigned int* counters) {
  constexpr int R = rows_per_warp(MT);
  dim3 grid((unsigned)ceil_div(a.N, WARPS * R), (unsigned)p.splits);
  const size_t smem = (size_t)MT * p.k_per_split * sizeof(float);
  // L2 budget of the early prefetch: about 32 MB over the whole grid
  const int64_t rows = (int64_t)grid.x * WARPS * R * p.splits;
  const int64_t prefetch = std::max<int64_t>(0, (int64_t(32) << 20) / std::max<int64_t>(rows, 1));
  return launch_pdl(gemv_kernel<MT, R>, grid, dim3(THREADS), smem, a.stream, a.out, a.a, a.w, a.c, part, counters,
                    (int)a.M, a.K, a.N, p.k_per_split, p.splits, prefetch);
}

// Resident blocks per SM of the decode kernel for MT rows and a K-slice of ks (cached).
int blocks_per_sm(int mt, int64_t ks) {
  static std::mutex mu;
  static int cache[64][5][128] = {{{0}}};  // device, log2(mt), ks / 128 (ks <= 12000 / mt)
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  const int mi = mt == 1 ? 0 : mt == 2 ? 1 : mt == 4 ? 2 : mt == 8 ? 3 : 4;
  const int ki = (int)std::min<int64_t>(127, ks / 128);
  std::lock_guard<std::mutex> lock(mu);
  int& v = cache[dev][mi][ki];
  if (v == 0) {
    const size_t smem = (size_t)mt * ks * sizeof(float);
    int n = 0;
    cudaError_t e = cudaErrorInvalidValue;
    switch (mt) {
      case 1: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemv_kernel<1, rows_per_warp(1)>, THREADS, smem); break;
      case 2: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemv_kernel<2, rows_per_warp(2)>, THREADS, smem); break;
      case 4: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemv_kernel<4, rows_per_warp(4)>, THREADS, smem); break;
      case 8: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemv_kernel<8, rows_per_warp(8)>, THREADS, smem); break;
      default: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemv_kernel<16, rows_per_warp(16)>, THREADS, smem);
    }
    if (e != cudaSuccess) cudaGetLastError();
    v = (e == cudaSuccess && n > 0) ? n : 1;
  }
  return v;
}

}  // namespace

int64_t gemv_max_ks(int64_t M) { return (SMEM_FLOATS / padded_m(M)) / 128 * 128; }

// K-split of the decode kernel: the number of splits s minimises waves(s) x (K/s + F), waves
// counting the resident block slots of all SMs, with K/s a multiple of 128 that fits the shared-
// memory slice and at least 256; F (the fixed cost of a block -- staging X~, the warp reduction,
// the split-K reduction -- in units of K) measured on GB300.
constexpr double kGemvFixedK = 512.0;

Plan plan_gemv(int64_t M, int64_t K, int64_t N, int sms) {
  Plan p{};
  p.kernel = kKernelGemv;
  const int mt = padded_m(M);
  const int64_t ks_max = (SMEM_FLOATS / mt) / 128 * 128;
  const int64_t groups = ceil_div(N, WARPS * rows_per_warp(mt));
  const int64_t s_min = ceil_div(K, ks_max);
  const int64_t s_max = std::max<int64_t>(s_min, std::min<int64_t>(64, K / 256));
  double best = 1e300;
  for (int64_t s = s_min; s <= s_max; ++s) {
    const int64_t ks = std::min<int64_t>(round_up(ceil_div(K, s), 128), ks_max);
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

spl_status run_gemv(const LinearArgs& a, const Plan& p) {
  if (p.splits > 65535) return SPL_ESHAPE;
  float* part = nullptr;
  unsigned int* counters = nullptr;
  if (p.splits > 1) {
    if (ceil_div(a.N, WARPS * rows_per_warp(padded_m(a.M))) > kMaxCounters) return SPL_ESHAPE;
    counters = static_cast<unsigned int*>(a.ws);
    part = reinterpret_cast<float*>(static_cast<char*>(a.ws) + kCounterBytes);
  }
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

// Device address of g_static_scratch on the current device.  The first call on
// a device looks it up (cudaGetSymbolAddress, with that device current) and
// clears the counter region; later calls reuse the cached address.
spl_status static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return SPL_ECUDA;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return SPL_ECUDA;
    if (cudaMemset(p, 0, kCounterBytes) != cudaSuccess) return SPL_ECUDA;
    g_static_ptr[dev] = p;
  }
  *out = g_static_ptr[dev];
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
  if (plan.splits > 1 && ceil_div(N, WARPS * rows_per_warp(padded_m(M))) > kMaxCounters) return SPL_EWORKSPACE;
  void* ws = nullptr;
  spl_status st = static_scratch(&ws);
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
  args.path = SPL_PATH_FP32;
  return run_gemv(args, plan);
}
