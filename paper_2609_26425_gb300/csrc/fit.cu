// fit.cu -- k-means centroids of one chunk per head (Sec. 2: the
// centroid-residual form of QVG with centroids kept in BF16, App. D.1).
//
// Lloyd iterations: initial centroid j = token floor(j*N/C); each iteration
// assigns every token to its Euclidean-nearest centroid (distance summed in
// channel order in fp32 with explicitly rounded operations, ties to the lower
// index) and replaces each non-empty cluster by its member mean (member sums
// accumulated in fp64, which is exact for bf16 members of ordinary range, so
// the result does not depend on the order of the atomic adds).
#include <mutex>

#include "qwm_internal.cuh"

namespace qwm {
namespace {

constexpr int FT = 128;  // tokens per assign CTA

__global__ void fit_init_kernel(const FitArgs a) {
  const int64_t n = (int64_t)a.H * a.C * a.d;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int c = (int)(i % a.d);
    const int j = (int)((i / a.d) % a.C);
    const int h = (int)(i / ((int64_t)a.d * a.C));
    const int64_t src = ((int64_t)j * a.N) / a.C;
    a.cent[i] = __bfloat162float(a.x[(src * a.H + h) * a.d + c]);
  }
}

__global__ void __launch_bounds__(FT) fit_assign_kernel(const FitArgs a) {
  extern __shared__ float sx[];  // [FT][d + 1]
  const int h = blockIdx.y;
  const int d = a.d, C = a.C;
  const int64_t t0 = (int64_t)blockIdx.x * FT;
  const int ld = d + 1;
  for (int i = threadIdx.x; i < FT * d; i += FT) {
    const int ti = i / d, c = i % d;
    const int64_t t = t0 + ti;
    sx[ti * ld + c] = t < a.N ? __bfloat162float(a.x[(t * a.H + h) * d + c]) : 0.0f;
  }
  __syncthreads();
  const int64_t t = t0 + threadIdx.x;
  if (t >= a.N) return;
  const float* xr = sx + threadIdx.x * ld;
  const float* mu = a.cent + (size_t)h * C * d;
  float best = 0.0f;
  int bj = -1;
  for (int j = 0; j < C; ++j) {
    const float* m = mu + (size_t)j * d;
    float acc = 0.0f;
    for (int c = 0; c < d; ++c) {
      const float tt = __fsub_rn(xr[c], __ldg(m + c));
      acc = __fadd_rn(acc, __fmul_rn(tt, tt));
    }
    if (bj < 0 || acc < best) { best = acc; bj = j; }
  }
  atomicAdd(a.counts + (size_t)h * C + bj, 1u);
  double* sum = a.sums + ((size_t)h * C + bj) * d;
  for (int c = 0; c < d; ++c) atomicAdd(sum + c, (double)xr[c]);
}

__global__ void fit_update_kernel(const FitArgs a) {
  const int64_t n = (int64_t)a.H * a.C * a.d;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t cnt = a.counts[i / a.d];
    if (cnt) a.cent[i] = __double2float_rn(__ddiv_rn(a.sums[i], (double)cnt));
  }
}

__global__ void fit_out_kernel(const FitArgs a) {
  const int64_t n = (int64_t)a.H * a.C * a.d;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    a.out[i] = __float2bfloat16_rn(a.cent[i]);
}

}  // namespace

size_t fit_workspace_bytes(int H, int d, int C) {
  const size_t hcd = (size_t)H * C * d;
  return (size_t)round_up(hcd * 4, 256) + (size_t)round_up(hcd * 8, 256) + (size_t)round_up((size_t)H * C * 4, 256);
}

cudaError_t launch_fit(const FitArgs& a, cudaStream_t st) {
  const int64_t n = (int64_t)a.H * a.C * a.d;
  const int eb = 256;
  const unsigned eg = (unsigned)((n + eb - 1) / eb < 4096 ? (n + eb - 1) / eb : 4096);
  fit_init_kernel<<<eg, eb, 0, st>>>(a);
  const size_t smem = (size_t)FT * (a.d + 1) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(fit_assign_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((a.N + FT - 1) / FT), (unsigned)a.H);
  for (int it = 0; it < a.iters; ++it) {
    if ((e = cudaMemsetAsync(a.sums, 0, (size_t)n * sizeof(double), st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.counts, 0, (size_t)a.H * a.C * sizeof(uint32_t), st)) != cudaSuccess) return e;
    fit_assign_kernel<<<grid, FT, smem, st>>>(a);
    fit_update_kernel<<<eg, eb, 0, st>>>(a);
  }
  fit_out_kernel<<<eg, eb, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace qwm

namespace qwm {

// ----------------------------------------------------------------------------
// Allocation-free variant of qwm_fit_centroids.
//
// Some callers cannot hand the library a scratch buffer: a plain C host
// program that only owns the input and output tensors it was given, or an
// inference engine whose device memory is already reserved by its own pool
// and which must not call cudaMalloc/cudaFree in the middle of generation
// (those calls can synchronise the whole device).  For them the k-means
// scratch (fp32 centroids, fp64 member sums, member counts) lives in this
// file-scope device array instead.
// ----------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocFitScratchBytes = (size_t)16 << 20;  // 16 MiB per GPU that loads the library
static __device__ __align__(256) uint8_t g_fit_scratch[kNoAllocFitScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_fit_scratch_mutex;
void* g_fit_scratch_addr[kMaxDevices] = {};

bool noalloc_cfg_ok(const qwm_config* c) {
  return c->num_heads >= 1 && c->num_heads <= 4096 && c->head_dim == kHeadDim &&
         (c->group_size == 32 || c->group_size == 64) && c->num_centroids >= 1 && c->num_centroids <= 256 &&
         (c->psac_rank == 0 || c->psac_rank == 8 || c->psac_rank == 16 || c->psac_rank == 32) &&
         c->num_candidates >= 1 && c->kmeans_iters >= 0;
}

}  // namespace
}  // namespace qwm

extern "C" QWM_API qwm_status qwm_fit_centroids_noalloc(const qwm_config* cfg, const void* x, int64_t N,
                                                        void* centroids, void* stream) {
  using namespace qwm;
  if (!cfg || !x || !centroids || N < 1) return QWM_ERR_INVALID_ARG;
  if (!noalloc_cfg_ok(cfg)) return QWM_ERR_UNSUPPORTED;
  if (N > (int64_t)1 << 31) return QWM_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) || (reinterpret_cast<uintptr_t>(centroids) & 15u))
    return QWM_ERR_INVALID_ARG;
  const size_t need = fit_workspace_bytes(cfg->num_heads, cfg->head_dim, cfg->num_centroids);
  if (need > kNoAllocFitScratchBytes) return QWM_ERR_CAPACITY;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return QWM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return QWM_ERR_UNSUPPORTED;
  uint8_t* ws = nullptr;
  {
    // First call on a device: look up the device address of the array there
    // (in host code its name is only a host-side stand-in).
    std::lock_guard<std::mutex> lock(g_fit_scratch_mutex);
    if (!g_fit_scratch_addr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_fit_scratch) != cudaSuccess || !p) return QWM_ERR_CUDA;
      g_fit_scratch_addr[dev] = p;
    }
    ws = static_cast<uint8_t*>(g_fit_scratch_addr[dev]);
  }
  FitArgs a{};
  a.H = cfg->num_heads; a.d = cfg->head_dim; a.C = cfg->num_centroids; a.iters = cfg->kmeans_iters;
  a.N = N;
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.out = static_cast<__nv_bfloat16*>(centroids);
  const size_t hcd = (size_t)a.H * a.C * a.d;
  a.cent = reinterpret_cast<float*>(ws);
  a.sums = reinterpret_cast<double*>(ws + round_up(hcd * 4, 256));
  a.counts = reinterpret_cast<uint32_t*>(ws + round_up(hcd * 4, 256) + round_up(hcd * 8, 256));
  // launch_fit writes every centroid before reading it and clears the sums
  // and counts before each iteration, so nothing depends on what an earlier
  // call left in the array.
  return launch_fit(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

