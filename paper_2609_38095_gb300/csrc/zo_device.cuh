// zo_device.cuh -- launch structures and device helpers shared by the kernels
// of the 1.5-SPSA parameter-space step (sm_103a).
#pragma once

#include <cstdint>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

namespace zo {

// Tensors described by one launch. The whole table travels in the kernel's
// parameter space (a 32 KB limit), so the library never allocates device
// memory for it; longer lists are split over several launches.
constexpr int kMaxTensorsPerLaunch = 1024;
constexpr int kMaxProbes = 1024;      // must match ZO_MAX_PROBES
constexpr int kMaxGroups = kMaxProbes / 8;

// Storage codes (match zo_dtype) and the per-tensor "vector path" flag.
constexpr uint8_t kF32 = 0, kBF16 = 1, kF16 = 2;
constexpr uint8_t kDtypeMask = 0x3;
constexpr uint8_t kVec32 = 0x80;      // base pointer is 32-byte aligned

// Elements are addressed by a virtual index g: tensor t starts at a multiple
// of 16, so each 16-element Philox block lies inside one tensor. Blocks are
// the unit of work: block b covers g in [16 b, 16 b + 16).
struct TensorTable {
  int32_t n;            // tensors in this launch
  int32_t pad_;
  int64_t blk_begin;    // first virtual block of tensor 0
  int64_t blk_end[kMaxTensorsPerLaunch];  // one past the last block of tensor t
  uint64_t ptr[kMaxTensorsPerLaunch];
  int64_t numel[kMaxTensorsPerLaunch];
  uint8_t flags[kMaxTensorsPerLaunch];    // dtype | kVec32
};

// Philox4x32 round keys, expanded on the host from the 64-bit step seed:
// key of round r = (seed_lo + r * W0, seed_hi + r * W1) mod 2^32.
struct RoundKeys {
  uint32_t k0[10];
  uint32_t k1[10];
};

struct PerturbParams {
  TensorTable tab;
  RoundKeys keys;
  uint32_t probe;          // probe index k
  float scale;             // used when coef == nullptr
  const double* coef;      // optional: scale = fp32(coef_mul * coef[probe])
  double coef_mul;
  const int32_t* status;   // optional: skip everything unless *status == 0
};

struct UpdateParams {
  TensorTable tab;
  RoundKeys keys;
  const double* coef;      // K coefficients c_k (device)
  double coef_mul;         // -(lr / K)
  int32_t K;
  int32_t groups;          // ceil(K / 8)
  const int32_t* status;   // optional
};

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11): ten rounds of two 32x32->64 products;
// the high halves are xored with the other two counter words and the round
// key, the low halves pass through. Round keys come from parameter space so
// they feed the xors without extra instructions.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                          const RoundKeys& rk) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t pa = static_cast<uint64_t>(0xD2511F53u) * c0;
    const uint64_t pb = static_cast<uint64_t>(0xCD9E8D57u) * c2;
    const uint32_t n0 = static_cast<uint32_t>(pb >> 32) ^ c1 ^ rk.k0[r];
    const uint32_t n2 = static_cast<uint32_t>(pa >> 32) ^ c3 ^ rk.k1[r];
    c1 = static_cast<uint32_t>(pb);
    c3 = static_cast<uint32_t>(pa);
    c0 = n0;
    c2 = n2;
  }
  return make_uint4(c0, c1, c2, c3);
}

__device__ __forceinline__ uint32_t word_of(const uint4& x, int m) {
  return m == 0 ? x.x : (m == 1 ? x.y : (m == 2 ? x.z : x.w));
}

// 256-bit global accesses (sm_100+): one per 16-element block of a 16-bit
// tensor, two for fp32. The caller guarantees 32-byte alignment.
#ifndef ZO_LDQ
#define ZO_LDQ ""  // cache qualifier of the streaming loads
#endif
#ifndef ZO_STQ
#define ZO_STQ ""  // cache qualifier of the streaming stores
#endif

__device__ __forceinline__ void ld256(const void* p, uint32_t (&r)[8]) {
  asm volatile("ld.global" ZO_LDQ ".v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "l"(p));
}

__device__ __forceinline__ void st256(void* p, const uint32_t (&r)[8]) {
  asm volatile("st.global" ZO_STQ ".v8.u32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(r[0]), "r"(r[1]), "r"(r[2]),
               "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
               : "memory");
}

// Widen / round 16-bit storage. A 32-bit register holds elements 2r (low
// half) and 2r + 1 (high half).
template <uint8_t DT>
__device__ __forceinline__ float2 unpack2(uint32_t u) {
  if constexpr (DT == kBF16) {
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xFFFF0000u));
  } else {
    __half2 h = *reinterpret_cast<__half2*>(&u);
    return __half22float2(h);
  }
}

template <uint8_t DT>
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  if constexpr (DT == kBF16) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
  } else {
    __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
  }
}

// Scalar element access for the element-wise path.
__device__ __forceinline__ float load_elem(const void* base, uint8_t dt, int64_t i) {
  if (dt == kF32) return static_cast<const float*>(base)[i];
  const uint16_t h = static_cast<const uint16_t*>(base)[i];
  if (dt == kBF16) return __uint_as_float(static_cast<uint32_t>(h) << 16);
  return __half2float(__ushort_as_half(h));
}

__device__ __forceinline__ void store_elem(void* base, uint8_t dt, int64_t i, float v) {
  if (dt == kF32) {
    static_cast<float*>(base)[i] = v;
  } else if (dt == kBF16) {
    static_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(v);
  } else {
    static_cast<__half*>(base)[i] = __float2half_rn(v);
  }
}

// Tensor containing virtual block b, searched forward from `t` (blocks of a
// thread only increase). Zero-length tensors own no block and are skipped.
__device__ __forceinline__ int advance_tensor(const TensorTable& tab, int t, int64_t b) {
  while (b >= tab.blk_end[t]) ++t;
  return t;
}

__device__ __forceinline__ int64_t tensor_blk_begin(const TensorTable& tab, int t) {
  return t == 0 ? tab.blk_begin : tab.blk_end[t - 1];
}

}  // namespace zo
