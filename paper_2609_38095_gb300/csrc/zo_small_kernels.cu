// zo_small_kernels.cu -- the probe-space preconditioner (Sec. 4.1, Eqs. 3-4)
// and the fixed-order fp64 reduction behind the quadratic test loss.
#include <mutex>

#include <cuda_runtime.h>

#include "zo_device.cuh"
#include "zo_launch.h"

namespace zo {

// ---------------------------------------------------------------------------
// Preconditioner, one thread per probe, fp64 throughout:
//   curv_k = (L+ - 2 L0 + L-) / eps^2                        (Eq. 3)
//   w_k    = 1 / max(lambda_reg, |curv_k|^alpha)             (Eq. 4)
//   c_k    = w_k (L+ - L-) / (2 eps)   or   w_k (L+ - L0) / eps
// With kPrecondRelative, Eq. 4 takes the relative curvature curv_k / m,
// m = (1/K) sum_j |curv_j| (a fixed-order block sum; m = 0 gives ratio 0):
// one reading of the per-step curvature normalisation of Sec. 6.
// Every value is checked before any is written: one non-finite loss,
// curvature, normaliser or coefficient makes the block write
// ZO_ERR_NONFINITE and nothing else. One block of up to kMaxProbes threads.
// ---------------------------------------------------------------------------
__global__ void precondition_kernel(const double* __restrict__ losses, int K, double eps, double alpha,
                                    double lambda_reg, int flags, double* __restrict__ c, double* __restrict__ w,
                                    double* __restrict__ curv, int32_t* __restrict__ status) {
  __shared__ double warp_sums[kMaxProbes / 32];
  __shared__ double s_norm;
  const int k = threadIdx.x;
  const bool one_sided = (flags & kPrecondOneSided) != 0;
  const bool relative = (flags & kPrecondRelative) != 0;
  double lp = 0.0, lm = 0.0, l0 = 0.0, cv = 0.0;
  bool bad = false;
  if (k < K) {
    lp = losses[3 * k + 0];
    lm = losses[3 * k + 1];
    l0 = losses[3 * k + 2];
    cv = __ddiv_rn(__dadd_rn(__dsub_rn(lp, __dmul_rn(2.0, l0)), lm), __dmul_rn(eps, eps));
    bad = !isfinite(lp) || !isfinite(lm) || !isfinite(l0) || !isfinite(cv);
  }
  double r = cv;
  if (relative) {
    // m: |curv| summed by a fixed shuffle tree per warp, warps in index order
    double v = (k < K && !bad) ? fabs(cv) : 0.0;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v = __dadd_rn(v, __shfl_down_sync(0xFFFFFFFFu, v, off));
    if ((k & 31) == 0) warp_sums[k >> 5] = v;
    __syncthreads();
    if (k == 0) {
      double sum = 0.0;
      for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) sum = __dadd_rn(sum, warp_sums[i]);
      s_norm = __ddiv_rn(sum, static_cast<double>(K));
    }
    __syncthreads();
    const double m = s_norm;
    bad = bad || !isfinite(m);
    r = m > 0.0 ? __ddiv_rn(cv, m) : 0.0;
  }
  double wk = 0.0, ck = 0.0;
  if (k < K) {
    wk = __ddiv_rn(1.0, fmax(lambda_reg, pow(fabs(r), alpha)));
    const double g = one_sided ? __ddiv_rn(__dsub_rn(lp, l0), eps) : __ddiv_rn(__dsub_rn(lp, lm), __dmul_rn(2.0, eps));
    ck = __dmul_rn(wk, g);
    bad = bad || !isfinite(ck);
  }
  bad = __syncthreads_or(bad);
  if (k == 0) *status = bad ? static_cast<int32_t>(kStatusNonFinite) : 0;
  if (bad || k >= K) return;
  c[k] = ck;
  if (w != nullptr) w[k] = wk;
  if (curv != nullptr) curv[k] = cv;
}

// ---------------------------------------------------------------------------
// f = 1/2 sum_i a_i theta_i^2 in fp64. Stage 1: each block folds a grid-
// strided slice (thread-sequential, then a fixed shuffle tree, then warps in
// index order) into partial[blockIdx.x]. Stage 2: one block folds the
// partials the same way. For a given grid size the order never changes, so
// the result is bit-reproducible.
// ---------------------------------------------------------------------------
__device__ __forceinline__ double block_sum(double v, double* warp_sums) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = __dadd_rn(v, __shfl_down_sync(0xFFFFFFFFu, v, off));
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) warp_sums[wid] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0) {
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) s = __dadd_rn(s, warp_sums[i]);
  }
  return s;
}

__global__ void __launch_bounds__(256) quad_loss_partial_kernel(const float* __restrict__ theta,
                                                                 const float* __restrict__ a, int64_t n,
                                                                 double* __restrict__ partial) {
  __shared__ double warp_sums[8];
  double s = 0.0;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride) {
    const double th = theta[i];
    s = __dadd_rn(s, __dmul_rn(static_cast<double>(a[i]), __dmul_rn(th, th)));
  }
  const double bs = block_sum(s, warp_sums);
  if (threadIdx.x == 0) partial[blockIdx.x] = bs;
}

__global__ void __launch_bounds__(256) quad_loss_final_kernel(const double* __restrict__ partial, int np,
                                                               double* __restrict__ out) {
  __shared__ double warp_sums[8];
  double s = 0.0;
  for (int i = threadIdx.x; i < np; i += blockDim.x) s = __dadd_rn(s, partial[i]);
  const double bs = block_sum(s, warp_sums);
  if (threadIdx.x == 0) *out = __dmul_rn(0.5, bs);
}

cudaError_t launch_precondition(const double* losses, int K, double eps, double alpha, double lambda_reg,
                                int flags, double* c, double* w, double* curv, int32_t* status,
                                cudaStream_t stream) {
  const int threads = ((K + 31) / 32) * 32;
  precondition_kernel<<<1, threads, 0, stream>>>(losses, K, eps, alpha, lambda_reg, flags, c, w, curv, status);
  return cudaGetLastError();
}

cudaError_t launch_quadratic_loss(const float* theta, const float* a, int64_t n, double* out, double* partial,
                                  int max_partials, int num_sms, cudaStream_t stream) {
  const int threads = 256;
  int64_t want = (n + threads * 8 - 1) / (threads * 8);
  int64_t cap = static_cast<int64_t>(num_sms) * 4;
  if (cap > max_partials) cap = max_partials;
  int grid = static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
  quad_loss_partial_kernel<<<grid, threads, 0, stream>>>(theta, a, n, partial);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  quad_loss_final_kernel<<<1, threads, 0, stream>>>(partial, grid, out);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Allocation-free variant of the quadratic loss. The partial sums live in a
// fixed array compiled into the library (every device that loads the library
// holds it until the process exits) instead of a caller workspace. Host code
// cannot use the array's name as a device address, so its address is looked
// up once per device with cudaGetSymbolAddress, with that device current.
// One partial per 2048-element slice: n <= kStaticLossPartials * 2048. Every
// block overwrites its own partial before the final fold reads it, so nothing
// needs clearing between calls; calls that overlap on the GPU share the array
// and race.
// ---------------------------------------------------------------------------
static __device__ __align__(256) double g_static_loss_partials[kStaticLossPartials];

namespace {
constexpr int kStaticMaxDevices = 64;
std::mutex g_static_mu;
double* g_static_ptr[kStaticMaxDevices] = {};
}  // namespace

cudaError_t static_loss_scratch(double** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kStaticMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (g_static_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_loss_partials);
    if (e != cudaSuccess) return e;
    g_static_ptr[dev] = static_cast<double*>(p);
  }
  *out = g_static_ptr[dev];
  return cudaSuccess;
}

cudaError_t launch_quadratic_loss_static(const float* theta, const float* a, int64_t n, double* out,
                                         cudaStream_t stream) {
  double* partial = nullptr;
  cudaError_t e = static_loss_scratch(&partial);
  if (e != cudaSuccess) return e;
  const int threads = 256;
  const int64_t want = (n + kStaticLossSlice - 1) / kStaticLossSlice;
  const int grid = static_cast<int>(want < 1 ? 1 : want);  // n is checked against the capacity by the caller
  quad_loss_partial_kernel<<<grid, threads, 0, stream>>>(theta, a, n, partial);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  quad_loss_final_kernel<<<1, threads, 0, stream>>>(partial, grid, out);
  return cudaGetLastError();
}

}  // namespace zo
