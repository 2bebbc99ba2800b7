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

// ---------------------------------------------------------------------------
// One forward point of the small quadratic workload in one pass: nops (0, 1
// or 2) perturbations of theta, applied exactly as zo_perturb / zo_perturb2
// apply them to an fp32 tensor (one fp32 add each), then the loss
// f(theta') = 1/2 sum a_i theta'_i^2 of the perturbed weights (Algorithm 1's
// ApplyPackedPerturbation followed by the forward pass, which for this
// workload is the reduction itself).
//
// A thread owns whole 16-element Philox blocks (grid-stride; theta is the
// parameter list's only tensor, so element i has virtual index i). Each term
// a_i theta_i^2 is formed without rounding as a pair of fp32 values
// (Dekker's exact product by fused multiply-add: a t = p + pe, p t = q + qe,
// term = q + fma(pe, t, qe), the last add carrying a relative error of about
// 2^-48) and summed into the thread's fp32 pair (s, sl) with Knuth's exact
// two-sum. Terms outside the range where those products are exact
// (|p| or |q| below 2^-100 or from 2^126 up, infinities, NaN) are added in
// fp64 instead, as (double)a * ((double)t * (double)t), behind a branch that
// is rarely taken: the fp64 pipe is slow on this GPU, and a predicated-off
// fp64 instruction still occupies it, so the loss above (five fp64
// operations per weight) takes 17 us on 2^20 weights. The pairs are summed
// over each warp's shuffle tree and converted to fp64 per warp, the warps
// added in order into one partial per CTA; the CTA that finishes last (a
// ticket counter in the workspace, reset by that CTA) folds the partials in
// index order and writes the result to out[j * out_stride], j < out_copies.
// No CTA waits for another. For a given grid the order of every sum is
// fixed: bit-reproducible.
// ---------------------------------------------------------------------------
// theta + scale z for element i of a block, fp32 storage: the probe bit moved
// to the sign by a multiply (PerturbOp::mul), as in the streaming passes.
__device__ __forceinline__ float add_signed_mul_f32(float th, const uint4& x, int i, const PerturbOp& op) {
  return __fadd_rn(th, __uint_as_float(op.nscale_bits ^ ((word_of(x, i >> 2) * op.mul[i & 3]) & 0x80000000u)));
}

struct QuadPassParams {
  float* theta;
  const float* a;
  int64_t n;
  RoundKeys keys;
  PerturbOp op[2];
  double* partial;      // one per CTA
  uint32_t* ticket;     // zero before the launch; the last CTA zeroes it again
  double* out;
  int32_t out_copies;
  int64_t out_stride;
};

struct DsSum {  // s + sl, an unevaluated fp32 pair
  float s = 0.0f, sl = 0.0f;
};

// ds += (q + r) by Knuth's two-sum of ds.s and q; the rounding error and r
// go to the low part.
__device__ __forceinline__ void ds_add(DsSum& ds, float q, float r) {
  const float s = __fadd_rn(ds.s, q);
  const float bb = __fsub_rn(s, ds.s);
  const float e = __fadd_rn(__fsub_rn(ds.s, __fsub_rn(s, bb)), __fsub_rn(q, bb));
  ds.sl = __fadd_rn(ds.sl, __fadd_rn(e, r));
  ds.s = s;
}

// The term a t^2 as q + r (see above); false when it leaves the range where
// the fp32 products are exact (then q = r = 0 and the caller adds it in fp64).
// Branch-free: the slow fp64 pipe is only reached through the caller's
// rarely taken branch.
__device__ __forceinline__ bool quad_term_ds(float av, float t, float& q, float& r) {
  const float p = __fmul_rn(av, t);
  const float pe = __fmaf_rn(av, t, -p);      // a t - p, exact
  const float q0 = __fmul_rn(p, t);
  const float qe = __fmaf_rn(p, t, -q0);      // p t - q, exact
  const float ap = fabsf(p), aq = fabsf(q0);
  const bool ok = ap >= 0x1p-100f && ap < 0x1p126f && aq >= 0x1p-100f && aq < 0x1p126f;
  q = ok ? q0 : 0.0f;
  r = ok ? __fmaf_rn(pe, t, qe) : 0.0f;       // the term's low part
  return ok;
}

// Sum of the CTA's fp32 pairs and fp64 parts, in a fixed order: pairs over
// each warp's shuffle tree (lane l takes lane l + off), converted to fp64 per
// warp with the warp's fp64 parts (shuffled only when one is non-zero), then
// the warps in index order. Returns the sum in thread 0.
__device__ __forceinline__ double block_sum_ds(DsSum ds, double dsum, double* warp_sums) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    DsSum o;
    o.s = __shfl_down_sync(0xFFFFFFFFu, ds.s, off);
    o.sl = __shfl_down_sync(0xFFFFFFFFu, ds.sl, off);
    ds_add(ds, o.s, o.sl);
  }
  if (__any_sync(0xFFFFFFFFu, dsum != 0.0)) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) dsum = __dadd_rn(dsum, __shfl_down_sync(0xFFFFFFFFu, dsum, off));
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) warp_sums[wid] = __dadd_rn(__dadd_rn(static_cast<double>(ds.s), static_cast<double>(ds.sl)), dsum);
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0) {
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) s = __dadd_rn(s, warp_sums[i]);
  }
  return s;
}

template <int NOPS, bool VEC>
__global__ void __launch_bounds__(256) perturb_quad_loss_kernel(const __grid_constant__ QuadPassParams P) {
  __shared__ double warp_sums[8];
  __shared__ bool last_s;
  DsSum ds;
  double dsum = 0.0;
  const int64_t nb = (P.n + 15) / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const bool same_ctr = P.op[1].ctr2 == P.op[0].ctr2;
  for (int64_t b = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; b < nb; b += stride) {
    const int64_t e0 = b * 16;
    const int cnt = static_cast<int>(min(static_cast<int64_t>(16), P.n - e0));
    float t[16], av[16];
    if (VEC && cnt == 16) {
      const float4* tp = reinterpret_cast<const float4*>(P.theta + e0);
      const float4* ap = reinterpret_cast<const float4*>(P.a + e0);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float4 x = tp[j], y = ap[j];
        t[4 * j] = x.x; t[4 * j + 1] = x.y; t[4 * j + 2] = x.z; t[4 * j + 3] = x.w;
        av[4 * j] = y.x; av[4 * j + 1] = y.y; av[4 * j + 2] = y.z; av[4 * j + 3] = y.w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        t[i] = i < cnt ? P.theta[e0 + i] : 0.0f;
        av[i] = i < cnt ? P.a[e0 + i] : 0.0f;
      }
    }
    if (NOPS >= 1) {
      const uint4 x0 = block_bits(b, P.op[0].ctr2, P.keys);
      uint4 x1 = x0;
      if (NOPS == 2 && !same_ctr) x1 = block_bits(b, P.op[1].ctr2, P.keys);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        t[i] = add_signed_mul_f32(t[i], x0, i, P.op[0]);
        if (NOPS == 2) t[i] = add_signed_mul_f32(t[i], x1, i, P.op[1]);
      }
      if (VEC && cnt == 16) {
        float4* tp = reinterpret_cast<float4*>(P.theta + e0);
#pragma unroll
        for (int j = 0; j < 4; ++j) tp[j] = make_float4(t[4 * j], t[4 * j + 1], t[4 * j + 2], t[4 * j + 3]);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (i < cnt) P.theta[e0 + i] = t[i];
      }
    }
    uint32_t wide = 0;  // terms that go to fp64
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float q, r;
      const bool ok = quad_term_ds(av[i], t[i], q, r);  // padding: a = t = 0, q = r = 0
      ds_add(ds, q, r);
      if (!ok && i < cnt) wide |= 1u << i;
    }
    if (wide != 0u) {
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if ((wide >> i) & 1u) {
          const double td = t[i];
          dsum = __dadd_rn(dsum, __dmul_rn(static_cast<double>(av[i]), __dmul_rn(td, td)));
        }
    }
  }
  const double bs = block_sum_ds(ds, dsum, warp_sums);
  if (threadIdx.x == 0) {
    P.partial[blockIdx.x] = bs;
    __threadfence();  // the partial is visible before the ticket counts it
    last_s = atomicAdd(P.ticket, 1u) == gridDim.x - 1u;
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();
  double s = 0.0;
  for (int i = threadIdx.x; i < static_cast<int>(gridDim.x); i += blockDim.x) s = __dadd_rn(s, __ldcg(P.partial + i));
  const double total = block_sum(s, warp_sums);
  if (threadIdx.x == 0) {
    const double f = __dmul_rn(0.5, total);
    for (int j = 0; j < P.out_copies; ++j) P.out[static_cast<int64_t>(j) * P.out_stride] = f;
    *P.ticket = 0u;
  }
}

cudaError_t launch_precondition(const double* losses, int K, double eps, double alpha, double lambda_reg,
                                int flags, double* c, double* w, double* curv, int32_t* status,
                                cudaStream_t stream) {
  const int threads = ((K + 31) / 32) * 32;
  precondition_kernel<<<1, threads, 0, stream>>>(losses, K, eps, alpha, lambda_reg, flags, c, w, curv, status);
  return cudaGetLastError();
}

cudaError_t launch_perturb_quad_loss(float* theta, const float* a, int64_t n, const RoundKeys& keys,
                                     const PerturbOp* ops, int nops, double* out, int out_copies, int64_t out_stride,
                                     double* partial, uint32_t* ticket, int max_partials, int num_sms,
                                     cudaStream_t stream) {
  QuadPassParams P;
  P.theta = theta;
  P.a = a;
  P.n = n;
  P.keys = keys;
  P.op[0] = ops[0];
  P.op[1] = nops == 2 ? ops[1] : ops[0];
  P.partial = partial;
  P.ticket = ticket;
  P.out = out;
  P.out_copies = out_copies;
  P.out_stride = out_stride;
  const int threads = 256;
  const int64_t want = ((n + 15) / 16 + threads - 1) / threads;
  int64_t cap = static_cast<int64_t>(num_sms) * 8;
  if (cap > max_partials) cap = max_partials;
  const int grid = static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
  const bool vec = reinterpret_cast<uintptr_t>(theta) % 16 == 0 && reinterpret_cast<uintptr_t>(a) % 16 == 0;
  switch (nops * 2 + (vec ? 1 : 0)) {
    case 0: perturb_quad_loss_kernel<0, false><<<grid, threads, 0, stream>>>(P); break;
    case 1: perturb_quad_loss_kernel<0, true><<<grid, threads, 0, stream>>>(P); break;
    case 2: perturb_quad_loss_kernel<1, false><<<grid, threads, 0, stream>>>(P); break;
    case 3: perturb_quad_loss_kernel<1, true><<<grid, threads, 0, stream>>>(P); break;
    case 4: perturb_quad_loss_kernel<2, false><<<grid, threads, 0, stream>>>(P); break;
    default: perturb_quad_loss_kernel<2, true><<<grid, threads, 0, stream>>>(P); break;
  }
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
