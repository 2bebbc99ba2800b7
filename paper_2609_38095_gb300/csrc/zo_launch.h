// zo_launch.h -- host-side launch wrappers shared between the kernel files and
// the C ABI layer (not part of the public interface).
#pragma once

#include <cuda_runtime.h>

#include "zo_device.cuh"

namespace zo {

constexpr int kStatusNonFinite = -4;  // ZO_ERR_NONFINITE
constexpr int kPrecondOneSided = 1;   // ZO_PRECOND_ONE_SIDED
constexpr int kPrecondRelative = 2;   // ZO_PRECOND_RELATIVE_CURVATURE
constexpr int kThreads = 256;         // threads per block of the streaming kernels
constexpr int kMaxLossPartials = 2048;
constexpr int kStaticLossPartials = 4096;   // fixed scratch of the allocation-free loss (32 KB)
constexpr int kMaxQuadPassPartials = 4096;  // CTAs of the one-pass perturbation + loss
constexpr int64_t kStaticLossSlice = 2048;  // elements per partial in that variant

// f32v: the launch holds 32-byte aligned fp32 tensors (single-op kernel only).
cudaError_t launch_perturb(const PerturbParams& p, int grid, int loop, bool f32v, cudaStream_t stream);
// dt: the storage type of the tensors grp_end counts (one launch per type).
cudaError_t launch_perturb_shift(const ShiftParams& p, uint8_t dt, int grid, cudaStream_t stream);
cudaError_t launch_perturb_pair(const PairParams& p, int grid, cudaStream_t stream);
// moved: theta at another offset from the 32-byte grid than plus and minus (16-bit only).
cudaError_t launch_pair_shift(const PairShiftParams& p, uint8_t dt, bool moved, int grid, cudaStream_t stream);
cudaError_t launch_update(const UpdateParams& p, int grid, cudaStream_t stream);
// Fused update with per-lane 8-probe tables (packing 1, up to 48 probe
// groups): one CTA of 512 threads per SM, two blocks per thread per chunk.
size_t lut8_smem_bytes(int groups);
bool lut8_supported(int groups, int packing);
cudaError_t lut8_prepare(int groups, int* blocks_per_sm);  // sets the shared-memory limit, occupancy
cudaError_t launch_update_lut8(const UpdateParams& p, int sms, int blocks_per_sm, cudaStream_t stream);
cudaError_t launch_update_shift(const UpdateShiftParams& p, uint8_t dt, int grid, cudaStream_t stream);
cudaError_t update_shift_blocks_per_sm(int groups, int packing, uint8_t dt, int* out);
size_t update_smem_bytes(int groups);
cudaError_t perturb_blocks_per_sm(int nops, int loop, int* out);
cudaError_t shift_blocks_per_sm(int nops, uint8_t dt, int* out);
cudaError_t pair_blocks_per_sm(int* out);
cudaError_t update_blocks_per_sm(int groups, int packing, int* out);
cudaError_t launch_probe_bytes(const RoundKeys& keys, uint32_t ctr2, uint32_t bit, int64_t first, int64_t n,
                               uint8_t* out, int grid, cudaStream_t stream);
cudaError_t launch_probe_signs(const RoundKeys& keys, uint32_t ctr2, uint32_t bit, int64_t first, int64_t n,
                               int8_t* out, int grid, cudaStream_t stream);
cudaError_t launch_precondition(const double* losses, int K, double eps, double alpha, double lambda_reg,
                                int flags, double* c, double* w, double* curv, int32_t* status,
                                cudaStream_t stream);
cudaError_t launch_quadratic_loss(const float* theta, const float* a, int64_t n, double* out, double* partial,
                                  int max_partials, int num_sms, cudaStream_t stream);
cudaError_t launch_quadratic_loss_static(const float* theta, const float* a, int64_t n, double* out,
                                         cudaStream_t stream);
// ops: nops (0, 1 or 2) perturbations; partial: max_partials doubles; ticket:
// a zeroed counter, zeroed again by the launch.
cudaError_t launch_perturb_quad_loss(float* theta, const float* a, int64_t n, const RoundKeys& keys,
                                     const PerturbOp* ops, int nops, double* out, int out_copies, int64_t out_stride,
                                     double* partial, uint32_t* ticket, int max_partials, int num_sms,
                                     cudaStream_t stream);

}  // namespace zo
