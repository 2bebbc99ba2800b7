/*
 * zo.h -- C ABI of the GB300 (sm_103a) parameter-space hot path of 1.5-SPSA,
 * "Probe-Space Preconditioning for Fast and Stable Zero-Order Training"
 * (Chaubard, Kochenderfer, Re).
 *
 * One training step of the method (Algorithm 1) touches the parameters only
 * through three operations, each one call here:
 *
 *   zo_perturb       theta <- theta + scale * z_k, in place        (Alg. 1; Sec. 4.3)
 *   zo_precondition  (L+, L-, L0) per probe -> coefficient c_k      (Sec. 4.1, Eqs. 3-4)
 *   zo_update        theta <- theta - (lr/K) * sum_k c_k z_k        (Sec. 4.2, Eqs. 5-6)
 *
 * plus a comparator, debug views of the probes and a reduction used by the
 * synthetic quadratic workload.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Memory. Every array argument is DEVICE memory of the current CUDA device,
 * owned by the caller, except the zo_tensor descriptor array itself (host
 * memory, read during the call only). The library allocates no device
 * memory: the tensor table travels inside the kernel launch parameters. Its
 * only CUDA objects are the timing events of zo_perturb2's launch
 * configuration choice (18 per parameter list, at most 64 lists, kept until
 * the process exits). Host side, each calling thread keeps its launch
 * parameter blocks (about 150 KB of thread-local storage).
 *
 * Streams. `stream` is a cudaStream_t (NULL = legacy default stream). Every
 * call only enqueues work on it and returns; results are visible to later
 * work on that stream. No call synchronises the device.
 *
 * Errors. Calls return a zo_status. Argument errors are detected on the host
 * before anything is enqueued. Launch failures return ZO_ERR_CUDA and the CUDA
 * message is available from zo_last_cuda_error() (per thread). Data-dependent
 * errors of the preconditioner are written to a device status word instead
 * (see zo_precondition). No call aborts or throws across the ABI.
 *
 * Parameter list. `params` is a list of n_tensors descriptors {ptr, numel,
 * dtype}: the trained weights, each updated in place. The same list, in the
 * same order and with the same sizes, must be given to every call of a step:
 * the probe is a function of the position of each element in that list.
 * Tensors may mix dtypes. numel may be 0 and at most 16 * (2^31 - 1) - 1
 * (ZO_ERR_ARG beyond). ptr must be aligned to its element size. Any such
 * alignment gives the same results; a tensor whose ptr is not 32-byte aligned
 * is streamed in 32-byte aligned chunks by a second kernel of the same call
 * (zo_perturb, zo_perturb2, zo_update, zo_update_ex, zo_update_sequential;
 * zo_perturb_pair when plus and minus share their offset), otherwise with
 * narrower accesses.
 *
 * Probes. z_k is Rademacher, one bit per parameter per probe (Sec. 2, Sec. 4.3
 * "Bit-Packed perturbations"; unpack rule of Appendix F: bit 1 -> +1, bit 0 ->
 * -1). It is never stored: it is regenerated from (seed, k, g) by the
 * counter-based generator Philox4x32-10 (Salmon et al., SC'11):
 *   g       virtual index of an element: tensor t starts at
 *           S_t = sum_{u<t} 16 * ceil(numel_u / 16), element i has g = S_t + i
 *   block   b = g / 16, probe group q = k / 8
 *   output  Philox4x32-10(counter = (b mod 2^32, b / 2^32, q, 0),
 *                         key = (seed mod 2^32, seed / 2^32)) = words x0..x3
 *   byte    m = g mod 16 is bits 8*(m mod 4) .. +7 of word x[m / 4]
 *   bit     z_k[g] = +1 if bit (k mod 8) of that byte is 1, else -1
 * so each 32-bit Philox word unpacks to four per-element bytes, each holding
 * the signs of eight probes ("packing 1": one generated bit per weight and
 * probe, as the paper's 1-bit packed perturbations).
 * With zo_set_packing(8) every (weight, probe) pair takes a whole generated
 * byte instead: output = Philox4x32-10(counter = (b mod 2^32, b / 2^32, k, 0),
 * key), byte m = g mod 16 as above, z_k[g] = +1 if bit 0 of that byte is 1.
 *
 * Arithmetic. Weights are read as fp32, the operation is done in fp32 and the
 * result is rounded once to the storage dtype (round to nearest even). A NaN
 * result is stored as the positive quiet NaN with every payload bit set
 * (0x7FFFFFFF fp32, 0x7FFF bf16 and fp16); infinities and signed zeros follow
 * IEEE 754.
 */
#ifndef ZO_H_
#define ZO_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { ZO_F32 = 0, ZO_BF16 = 1, ZO_F16 = 2 } zo_dtype;

typedef struct {
  void* ptr;     /* device pointer to the weights (contiguous)            */
  int64_t numel; /* number of elements, >= 0                              */
  int32_t dtype; /* zo_dtype                                              */
  int32_t reserved; /* must be 0                                          */
} zo_tensor;

typedef enum {
  ZO_OK = 0,
  ZO_ERR_ARG = -1,             /* null pointer, negative size, bad scalar      */
  ZO_ERR_DTYPE = -2,           /* unknown dtype code                           */
  ZO_ERR_ALIGN = -3,           /* pointer not aligned to its element size      */
  ZO_ERR_NONFINITE = -4,       /* a loss, curvature or coefficient not finite  */
  ZO_ERR_CUDA = -5,            /* a CUDA runtime call failed                   */
  ZO_ERR_TOO_MANY_PROBES = -6, /* K > ZO_MAX_PROBES                            */
  ZO_ERR_WORKSPACE = -7        /* workspace missing or too small               */
} zo_status;

/* Largest K accepted by zo_update / zo_update_sequential / zo_precondition. */
#define ZO_MAX_PROBES 1024

/* Human-readable name of a zo_status value (static storage). */
const char* zo_status_string(int status);

/* Message of the last CUDA error seen by a zo_* call on this thread ("" if none). */
const char* zo_last_cuda_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int zo_version(void);

/* Probe packing used by every later call of the process: 1 (default) or 8
 * generated bits per (weight, probe), see "Probes" above (Sec. 4.3 "Bit-Packed
 * perturbations" packs one bit; 8 gives each weight a whole byte per probe).
 * Set it before a step and keep it for the whole step: every call of a step
 * must regenerate the same probes. Returns ZO_ERR_ARG for other values. */
int zo_set_packing(int32_t bits_per_value);
int zo_get_packing(void);

/* ---------------------------------------------------------------------------
 * zo_perturb -- Algorithm 1, ApplyPackedPerturbation(theta, scale, z_k): adds
 * scale * z_k to every weight in place. A probe's forward passes call it with
 * scale = +eps, then -2 eps, then +eps to restore (Algorithm 1; Appendix F
 * "_unpack_and_apply" is the paper's version of this operation).
 *   params, n_tensors  the parameter list (see above); n_tensors >= 0
 *   seed               64-bit step seed
 *   probe              probe index k
 *   scale              fp32 amount; element result = rn(fp32(theta) + scale*z)
 * Errors: ZO_ERR_ARG, ZO_ERR_DTYPE, ZO_ERR_ALIGN, ZO_ERR_CUDA.
 * ------------------------------------------------------------------------- */
int zo_perturb(const zo_tensor* params, int32_t n_tensors, uint64_t seed, uint32_t probe, float scale,
               void* stream);

/* ---------------------------------------------------------------------------
 * zo_perturb2 -- two consecutive perturbations in one pass over theta:
 * exactly zo_perturb(probe_a, scale_a) followed by zo_perturb(probe_b,
 * scale_b) (each result rounded to storage, bit for bit the same), with one
 * read and one write of every weight instead of two. In Algorithm 1 no
 * forward pass runs between probe k's restore (+eps) and probe k+1's first
 * perturbation (+eps), so a step can apply them together:
 * zo_perturb2(k, +eps, k + 1, +eps). Errors as zo_perturb.
 * Launch configuration: the first nine calls on a parameter list (identified
 * by device, sizes, dtypes and 32-byte alignments) each run one of three
 * loop / grid configurations between two CUDA events recorded on `stream`;
 * later calls use the fastest. The results never depend on the
 * configuration. Calls made while `stream` is being captured into a CUDA
 * graph use the first configuration and record no event.
 * ------------------------------------------------------------------------- */
int zo_perturb2(const zo_tensor* params, int32_t n_tensors, uint64_t seed, uint32_t probe_a, float scale_a,
                uint32_t probe_b, float scale_b, void* stream);

/* zo_perturb_pair -- both forward points of probe k in one pass, out of place:
 *   plus  <- rn( fp32(theta) + scale * z_k )
 *   minus <- rn( fp32(theta) - scale * z_k )
 * for every tensor, theta left untouched (Sec. 2 / Eq. 3 evaluate the loss at
 * theta +- eps z; Algorithm 1 reaches them in place by +eps, -2 eps, +eps).
 * theta is read once and the two results written once: 6 bytes per 16-bit
 * weight instead of the 8 of two in-place passes, no restore pass and no
 * restore drift, for two extra copies of the weights in device memory.
 * The probes are zo_perturb's: `theta` is the parameter list of the step
 * (virtual indices from its sizes); plus and minus are lists of the same
 * length with the same numel and dtype per entry. plus[t] may be theta[t]
 * itself (then theta becomes theta + scale z) and so may minus[t]; plus[t]
 * and minus[t] must be different, and any other overlap is undefined.
 * Access paths (same results): 256-bit blocks when all three pointers of a
 * 16-bit tensor are 32-byte aligned; 32-byte aligned chunks when plus and
 * minus share their offset from that grid (theta at any offset) and for fp32
 * tensors whose three pointers share it; narrower accesses otherwise.
 * Errors: ZO_ERR_ARG (also for mismatched lists or plus[t] == minus[t]),
 * ZO_ERR_DTYPE, ZO_ERR_ALIGN, ZO_ERR_CUDA. No counterpart in the paper as a
 * kernel: it trades device memory for HBM traffic. */
int zo_perturb_pair(const zo_tensor* theta, const zo_tensor* plus, const zo_tensor* minus, int32_t n_tensors,
                    uint64_t seed, uint32_t probe, float scale, void* stream);

/* ---------------------------------------------------------------------------
 * zo_precondition -- the probe-space diagonal preconditioner of Sec. 4.1 with
 * the paper's settings (alpha = 0.1, lambda_reg = 1, two-sided difference).
 * For each probe k, from losses row k = {L+_k, L-_k, L0_k} (device, K x 3 fp64,
 * row-major):
 *   curv_k = (L+ - 2 L0 + L-) / eps^2                       (Eq. 3)
 *   w_k    = 1 / max(lambda_reg, |curv_k|^alpha)            (Eq. 4)
 *   c_k    = w_k * (L+ - L-) / (2 eps)                      (Eq. 5; Alg. 1 g_i w_i)
 *   c      device, K fp64, written only when every value is finite
 *   status device, one int32: ZO_OK, or ZO_ERR_NONFINITE when any loss,
 *          curvature or coefficient is NaN/Inf (then c is left untouched).
 * Host-side errors (nothing enqueued): ZO_ERR_ARG (K < 1, eps <= 0 or not
 * finite, null pointer), ZO_ERR_TOO_MANY_PROBES, ZO_ERR_CUDA.
 * ------------------------------------------------------------------------- */
int zo_precondition(const double* losses, int32_t K, double eps, double* c, int32_t* status, void* stream);

/* Bits of zo_precondition_ex's `flags` (0 = the paper's preconditioner). */
#define ZO_PRECOND_ONE_SIDED 1          /* c_k = w_k (L+ - L0) / eps, a non-paper forward difference */
#define ZO_PRECOND_RELATIVE_CURVATURE 2 /* Eq. 4 on curv_k / m, m = (1/K) sum_j |curv_j| */

/* zo_precondition with every knob of Sec. 4.1 exposed: alpha in [0, 1]
 * (alpha = 0 recovers 1SPSA, alpha = 1 is a diagonal Newton step in probe
 * space), lambda_reg > 0, and `flags`, a bitwise OR of:
 *   ZO_PRECOND_ONE_SIDED           the forward difference above instead of
 *                                  the paper's central one;
 *   ZO_PRECOND_RELATIVE_CURVATURE  Eq. 4 applied to the relative curvature
 *       r_k = curv_k / m with m = (1/K) sum_j |curv_j| over this call's K
 *       probes (r_k = 0 for all k when m = 0; a non-finite m is
 *       ZO_ERR_NONFINITE). Sec. 6 names per-step curvature normalisation as
 *       future work without a formula; this is one reading of it: the weight
 *       then depends only on how a probe's curvature compares with the
 *       step's average, not on the loss scale.
 * Any other bit is ZO_ERR_ARG. w and curv (device, K fp64) are optional
 * outputs (NULL to skip), written under the same rule as c; curv is always
 * Eq. 3's curvature. */
int zo_precondition_ex(const double* losses, int32_t K, double eps, double alpha, double lambda_reg,
                       int32_t flags, double* c, double* w, double* curv, int32_t* status, void* stream);

/* ---------------------------------------------------------------------------
 * zo_update -- the fused K-probe update of Sec. 4.2 (Eq. 5 and its compact form
 * Eq. 6, Delta theta = -eta Z W dl), in one read and one write of theta:
 *   a_k   = fp32( (-(lr / K)) * c_k )    (fp64 product, rounded to fp32)
 *   theta <- rn( fp32(theta) + sum_{k<K} a_k z_k )
 * with the sum accumulated in fp32, eight probes at a time in increasing
 * probe order: the partial of probes 8q..8q+7 is the fp32 sum of the 4-probe
 * partials ((s0 a0 + s1 a1) + s2 a2) + s3 a3 of probes 8q..8q+3 and of
 * 8q+4..8q+7 (s_j = z of that probe), and these 8-probe partials are added
 * to the running sum in increasing q (probes K..8*ceil(K/8)-1 have a = 0).
 * With lr = eps this is Algorithm 1's gamma_k = g_k w_k / (2n) step, fused
 * over all probes.
 *   c       device, K fp64 coefficients (normally zo_precondition's output)
 *   K       1 .. ZO_MAX_PROBES; probes 0..K-1 of `seed`
 *   lr      step size (the paper ties it to eps)
 *   status  optional device int32 (NULL to ignore): when it holds anything but
 *           ZO_OK at execution time the update leaves theta untouched.
 * Errors: ZO_ERR_ARG, ZO_ERR_DTYPE, ZO_ERR_ALIGN, ZO_ERR_TOO_MANY_PROBES,
 * ZO_ERR_CUDA.
 * ------------------------------------------------------------------------- */
int zo_update(const zo_tensor* params, int32_t n_tensors, uint64_t seed, const double* c, int32_t K, double lr,
              const int32_t* status, void* stream);

/* zo_update preceded, in the same pass, by one perturbation: exactly
 * zo_perturb(pre_probe, pre_scale) then zo_update(...) (the perturbed value
 * is rounded to storage before the probe sum is added), with one read and
 * one write of theta. Used to fold the last probe's restore (+eps) into the
 * update. has_pre = 0 makes it zo_update. When `status` holds anything but
 * ZO_OK only the leading perturbation is applied (a restore must always
 * happen). Errors as zo_update (ZO_ERR_ARG also for a non-finite pre_scale). */
int zo_update_ex(const zo_tensor* params, int32_t n_tensors, uint64_t seed, const double* c, int32_t K, double lr,
                 const int32_t* status, int32_t has_pre, uint32_t pre_probe, float pre_scale, void* stream);

/* Comparator with Algorithm 1's own schedule: K in-place passes, pass k adds
 * a_k z_k (same a_k as zo_update) and rounds to storage, exactly as
 * zo_perturb(scale = a_k). Same arguments and errors as zo_update. */
int zo_update_sequential(const zo_tensor* params, int32_t n_tensors, uint64_t seed, const double* c, int32_t K,
                         double lr, const int32_t* status, void* stream);

/* ---------------------------------------------------------------------------
 * Debug views of a probe (never needed by a training step).
 * zo_probe_bytes writes probe k packed one bit per element in the layout
 * Appendix F unpacks (element 8j+i is bit i of byte j), bytes first..first+n-1
 * of the virtual index space, to out (device, n bytes).
 * zo_probe_signs writes z_k[g] as int8 (+1 / -1) for g = first..first+n-1.
 * Errors: ZO_ERR_ARG (negative first/n, null out with n > 0), ZO_ERR_CUDA.
 * ------------------------------------------------------------------------- */
int zo_probe_bytes(uint64_t seed, uint32_t probe, int64_t first, int64_t n, uint8_t* out, void* stream);
int zo_probe_signs(uint64_t seed, uint32_t probe, int64_t first, int64_t n, int8_t* out, void* stream);

/* ---------------------------------------------------------------------------
 * zo_quadratic_loss -- f(theta) = 1/2 sum_i a_i theta_i^2 over n fp32 elements,
 * accumulated in fp64 in a fixed order (bit-reproducible for a given device),
 * written to out (device, one fp64). It stands in for the model forward of
 * Algorithm 1 on the small synthetic workload (an ill-conditioned quadratic
 * of the stiff-paraboloid family of Sec. 5.3).
 *   workspace  device scratch of at least zo_quadratic_loss_workspace_size(n)
 *              bytes, not shared with concurrent calls.
 * Errors: ZO_ERR_ARG, ZO_ERR_WORKSPACE, ZO_ERR_CUDA.
 * ------------------------------------------------------------------------- */
int64_t zo_quadratic_loss_workspace_size(int64_t n);
int zo_quadratic_loss(const float* theta, const float* a, int64_t n, double* out, void* workspace,
                      int64_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * zo_quadratic_loss_static -- zo_quadratic_loss for callers that cannot
 * allocate device memory. The paper has no counterpart: it exists for code
 * that runs inside a device-memory budget fixed in advance (for example a
 * framework whose caching allocator already holds the device memory, where
 * an extra cudaMalloc fails) or that must not let an allocation synchronise
 * the device (cudaMalloc and cudaFree may). It computes the same value as
 * zo_quadratic_loss without a workspace argument: its scratch is a fixed
 * 32 KB array inside the library, held by every device that loads the
 * library until the process exits. The call allocates nothing.
 *   n     0 .. ZO_QUADRATIC_LOSS_STATIC_MAX_N elements; larger n returns
 *         ZO_ERR_WORKSPACE (the fixed scratch holds one partial sum per 2048
 *         elements) and enqueues nothing.
 * The first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any stream
 * capture. All calls share the array: calls that overlap on the GPU (other
 * streams, other host threads on the same device) race and must be ordered
 * by the caller. Nothing in it needs clearing between calls.
 * Errors: ZO_ERR_ARG, ZO_ERR_WORKSPACE, ZO_ERR_CUDA.
 * ------------------------------------------------------------------------- */
#define ZO_QUADRATIC_LOSS_STATIC_MAX_N 8388608
int zo_quadratic_loss_static(const float* theta, const float* a, int64_t n, double* out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* ZO_H_ */
