// Row / column statistics of one matrix without any device allocation.
//
// Some callers cannot call cudaMalloc: code that runs inside a framework
// which owns all device memory through its own pool and forbids outside
// allocations, and latency-critical paths that must not allocate after
// start-up (cudaMalloc may synchronise the whole device). For them this file
// provides meq_row_col_stats_noalloc(), the statistics step of the optimizer
// (row / column RMS, their coefficients of variation and the chosen
// normalisation side) for one caller-provided matrix. Its scratch lives in a
// file-scope __device__ array of fixed size that every GPU which loads the
// library holds until the process exits.
//
// It sums squares over blocks of 32 rows x 1024 columns, folds the partials
// with one thread per row and per column (blocks in order), and forms the
// CVs in two passes, all in
// fp32 like the full step's statistics, so results agree with meq_read_stats
// up to fp32 summation order. The same kernels, given scratch that the caller
// allocated, give the first point of the CV trajectory (meq_ns_cv_trajectory).
#include <mutex>
#include <string>

#include "../../include/meq.h"
#include "meq_elementwise.cuh"

namespace {

constexpr int kNaThreads = 256;
constexpr int kNaSlab = 32;        // rows per block
constexpr int kNaChunk = 1024;     // columns per block (four per thread)
constexpr int kNaFoldThreads = 256;
constexpr int kNaFinThreads = 1024;
constexpr int kMaxDevices = 64;

// 8 MiB of scratch: the row partial sums of squares (ceil(cols / 1024) x
// rows floats) followed by the column partial sums (ceil(rows / 32) x cols).
constexpr long long kScratchFloats = 2ll * 1024 * 1024;
static __device__ __align__(256) float g_stats_scratch[kScratchFloats];

std::mutex g_setup_mu;
float* g_scratch_addr[kMaxDevices] = {nullptr};

__device__ __forceinline__ float na_block_sum_f32(float v, float* sh) {
  const unsigned FULL = 0xffffffffu;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) sh[w] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float r = 0.f;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) r += sh[i];
    sh[0] = r;
  }
  __syncthreads();
  return sh[0];
}

// One block per 32-row slab (blockIdx.x) and 1024-column chunk (blockIdx.y):
// the slab's column partial sums of squares over the chunk's columns, and
// the chunk's partial sums of squares of the slab's rows.
__global__ void __launch_bounds__(kNaThreads) na_stats_kernel(const float* __restrict__ U, int64_t m, int64_t n,
                                                              float* __restrict__ scratch) {
  __shared__ float shr[kNaThreads / 32][32];
  const int64_t slab = blockIdx.x, chunk = blockIdx.y;
  const int64_t r0 = slab * kNaSlab;
  const int nr = static_cast<int>(m - r0 < kNaSlab ? m - r0 : kNaSlab);
  const int64_t c1 = (chunk + 1) * kNaChunk < n ? (chunk + 1) * kNaChunk : n;
  const int64_t nchunks = (n + kNaChunk - 1) / kNaChunk;
  const float* Us = U + r0 * n;
  float* rowss = scratch + chunk * m;
  float* cp = scratch + nchunks * m + slab * n;
  float racc[kNaSlab];
#pragma unroll
  for (int r = 0; r < kNaSlab; ++r) racc[r] = 0.f;
  for (int64_t c = chunk * kNaChunk + threadIdx.x; c < c1; c += kNaThreads) {
    float cacc = 0.f;
#pragma unroll
    for (int r = 0; r < kNaSlab; ++r) {
      if (r < nr) {
        const float u = Us[r * n + c];
        const float u2 = u * u;
        cacc += u2;
        racc[r] += u2;
      }
    }
    cp[c] = cacc;
  }
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const bool up = (lane & o) != 0;
      const float send = up ? racc[i] : racc[i + o];
      const float keep = up ? racc[i + o] : racc[i];
      racc[i] = keep + __shfl_xor_sync(FULL, send, o);
    }
  }
  shr[w][lane] = racc[0];
  __syncthreads();
  if (threadIdx.x < nr) {
    float s = 0.f;
    for (int i = 0; i < kNaThreads / 32; ++i) s += shr[i][threadIdx.x];
    rowss[r0 + threadIdx.x] = s;
  }
}

// r (Eq. (7)) from the row partials and c from the column partials, one
// thread per row / column, each summing its partials in block order; the
// row sums of squares are kept (first row of the scratch) for the CV kernel.
__global__ void __launch_bounds__(kNaFoldThreads) na_fold_kernel(int64_t m, int64_t n, float* __restrict__ scratch,
                                                                 float* __restrict__ r, float* __restrict__ c) {
  const int64_t t = static_cast<int64_t>(blockIdx.x) * kNaFoldThreads + threadIdx.x;
  const int64_t nslabs = (m + kNaSlab - 1) / kNaSlab;
  const int64_t nchunks = (n + kNaChunk - 1) / kNaChunk;
  const float* cpart = scratch + nchunks * m;
  if (t < m) {
    float acc = 0.f;
    for (int64_t k = 0; k < nchunks; ++k) acc += scratch[k * m + t];
    scratch[t] = acc;  // only this thread reads or writes row t's partials
    r[t] = sqrtf(acc * (1.0f / static_cast<float>(n)));
  }
  if (t < n) {
    float acc = 0.f;
    int64_t k = 0;
    for (; k + 4 <= nslabs; k += 4) {  // four loads in flight, added in slab order
      const float a0 = cpart[k * n + t], a1 = cpart[(k + 1) * n + t];
      const float a2 = cpart[(k + 2) * n + t], a3 = cpart[(k + 3) * n + t];
      acc += a0;
      acc += a1;
      acc += a2;
      acc += a3;
    }
    for (; k < nslabs; ++k) acc += cpart[k * n + t];
    c[t] = sqrtf(acc * (1.0f / static_cast<float>(m)));
  }
}

// gamma_r, gamma_c (Eq. (8), over entries > delta) and the side (Eq. (11)),
// all fp32, in one block. With frob set, r and c are first divided by
// ||U||_F (from the row sums of squares, fixed order), so that they and the
// threshold describe X = U / ||U||_F; a zero U gives zeros.
__global__ void __launch_bounds__(kNaFinThreads) na_cv_kernel(int64_t m, int64_t n, float delta, float tie_atol, int frob,
                                                              const float* __restrict__ scratch, float* __restrict__ r,
                                                              float* __restrict__ c, double* __restrict__ gammas,
                                                              int* __restrict__ direction) {
  __shared__ float shf[32];
  if (frob) {
    float tot = 0.f;
    for (int64_t i = threadIdx.x; i < m; i += blockDim.x) tot += scratch[i];
    tot = na_block_sum_f32(tot, shf);
    const float inv = tot > 0.f ? 1.0f / sqrtf(tot) : 0.f;
    for (int64_t i = threadIdx.x; i < m; i += blockDim.x) r[i] *= inv;
    for (int64_t j = threadIdx.x; j < n; j += blockDim.x) c[j] *= inv;
    __syncthreads();
  }
  float gam[2];
  for (int side = 0; side < 2; ++side) {
    const float* v = side == 0 ? r : c;
    const int64_t len = side == 0 ? m : n;
    float cnt = 0.f, sum = 0.f;
    for (int64_t i = threadIdx.x; i < len; i += blockDim.x) {
      const float x = v[i];
      if (x > delta) cnt += 1.f, sum += x;
    }
    cnt = na_block_sum_f32(cnt, shf);
    sum = na_block_sum_f32(sum, shf);
    const float mean = cnt > 0.f ? sum / cnt : 0.f;
    float var = 0.f;
    for (int64_t i = threadIdx.x; i < len; i += blockDim.x) {
      const float x = v[i];
      if (x > delta) var += (x - mean) * (x - mean);
    }
    var = na_block_sum_f32(var, shf);
    gam[side] = cnt > 0.f ? sqrtf(var / cnt) / mean : 0.f;
  }
  if (threadIdx.x == 0) {
    gammas[0] = static_cast<double>(gam[0]);
    gammas[1] = static_cast<double>(gam[1]);
    *direction = gam[0] >= gam[1] - tie_atol ? 0 : 1;
  }
}

// Plain launch (no attributes) that returns this launch's own status.
template <typename... KArgs, typename... Args>
cudaError_t launch_plain(void (*kernel)(KArgs...), dim3 grid, unsigned block, cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(block);
  cfg.stream = st;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Device address of the scratch array on the current device, looked up once
// per device (the host-side symbol is only a stand-in, not a device address).
cudaError_t scratch_address(float** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_stats_scratch);
    if (e != cudaSuccess) return e;
    if (p == nullptr) return cudaErrorInvalidSymbol;
    g_scratch_addr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

meq_status na_fail(meq_status s, const std::string& msg) {
  meq::set_global_error(msg);
  return s;
}

}  // namespace

namespace meq {

int64_t row_col_stats_scratch_floats(int64_t rows, int64_t cols) {
  return (cols + kNaChunk - 1) / kNaChunk * rows + (rows + kNaSlab - 1) / kNaSlab * cols;
}

cudaError_t launch_row_col_stats(const float* U, int64_t rows, int64_t cols, float eps, float tie_atol, int frob,
                                 float* scratch, float* r, float* c, double* gammas, int* direction, cudaStream_t st,
                                 const char** failed) {
  const int64_t nslabs = (rows + kNaSlab - 1) / kNaSlab;
  const int64_t nchunks = (cols + kNaChunk - 1) / kNaChunk;
  *failed = "statistics launch";
  cudaError_t e = launch_plain(na_stats_kernel, dim3(static_cast<unsigned>(nslabs), static_cast<unsigned>(nchunks)),
                               kNaThreads, st, U, rows, cols, scratch);
  if (e != cudaSuccess) return e;
  *failed = "fold launch";
  const int64_t len = rows > cols ? rows : cols;
  e = launch_plain(na_fold_kernel, dim3(static_cast<unsigned>((len + kNaFoldThreads - 1) / kNaFoldThreads)),
                   kNaFoldThreads, st, rows, cols, scratch, r, c);
  if (e != cudaSuccess) return e;
  *failed = "CV launch";
  return launch_plain(na_cv_kernel, dim3(1), kNaFinThreads, st, rows, cols, eps, tie_atol, frob,
                      static_cast<const float*>(scratch), r, c, gammas, direction);
}

}  // namespace meq

extern "C" meq_status meq_row_col_stats_noalloc(const float* U, int64_t rows, int64_t cols, float eps, float tie_atol,
                                                float* r, float* c, double* gammas, int* direction,
                                                void* cuda_stream) {
  if (!U || !r || !c || !gammas || !direction)
    return na_fail(MEQ_ERR_INVALID_ARG, "meq_row_col_stats_noalloc: U, r, c, gammas and direction must not be NULL");
  if (rows <= 0 || cols <= 0 || rows > (int64_t(1) << 20) || cols > (int64_t(1) << 20))
    return na_fail(MEQ_ERR_INVALID_ARG, "meq_row_col_stats_noalloc: rows and cols must be in 1..2^20");
  if (!(eps >= 0.f) || !(tie_atol >= 0.f))
    return na_fail(MEQ_ERR_INVALID_ARG, "meq_row_col_stats_noalloc: eps and tie_atol must be >= 0");
  const int64_t need = meq::row_col_stats_scratch_floats(rows, cols);
  if (need > kScratchFloats)
    return na_fail(MEQ_ERR_INVALID_ARG, "meq_row_col_stats_noalloc: " + std::to_string(rows) + " x " +
                                            std::to_string(cols) + " needs " + std::to_string(need) +
                                            " floats of scratch, above the fixed " + std::to_string(kScratchFloats));
  float* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess)
    return na_fail(MEQ_ERR_CUDA, std::string("meq_row_col_stats_noalloc: scratch address lookup: ") + cudaGetErrorString(e));
  const char* what = "";
  e = meq::launch_row_col_stats(U, rows, cols, eps, tie_atol, 0, scratch, r, c, gammas, direction,
                                static_cast<cudaStream_t>(cuda_stream), &what);
  if (e != cudaSuccess)
    return na_fail(MEQ_ERR_CUDA, std::string("meq_row_col_stats_noalloc: ") + what + ": " + cudaGetErrorString(e));
  return MEQ_OK;
}
