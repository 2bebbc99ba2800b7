// zo_update_lut8.cu -- the fused K-probe update (Sec. 4.2, Eqs. 5-6) with one
// table lookup per eight probes.
//
// theta <- rn(fp32(theta) + sum_k a_k z_k[g]), a_k = fp32(coef_mul * c_k).
//
// Byte m of Philox(b, q) carries the signs of probes 8q..8q+7 of element
// 16b + m (packing 1). For each probe group q the 256-entry table
//   T8_q[n] = T_lo[n & 15] + T_hi[n >> 4],
//   T_lo[i] = ((s0 a_{8q} + s1 a_{8q+1}) + s2 a_{8q+2}) + s3 a_{8q+3}  (s_j = +1 iff bit j of i)
// and T_hi likewise for probes 8q+4..8q+7, holds the group's fp32 partial sum
// for every sign byte n. An element adds one looked-up value per group, groups
// in increasing order: one byte-permute (the address), one shared load and
// half a packed fp32x2 add per eight probes. update_kernel adds exactly these
// partials in this order (as two 4-probe lookups), so the two kernels give
// the same bits.
//
// Bank conflicts. 32 lanes looking up random bytes of one 256-entry table
// would collide on the 32 shared-memory banks, so every lane reads its own
// copy: row n of the replicated region (256 bytes) holds T8[n] once per lane,
// lane l in word l of one half of the row (bank l), and another group's table
// in the other half. The lookup address is then
//   region + 256 n + 128 h + 4 l,
// with the region on a 64 KB boundary of the shared window: one byte-permute
// puts the sign byte n under the region's upper half-word and next to the
// lane's offset 128 h + 4 l.
//
// Loop order. The replicated tables of all groups do not fit in shared memory
// (32 KB per group), so probe groups are the outer loop: a CTA owns a chunk of
// 512 * BPT consecutive blocks (BPT = 8 on large launches), accumulates every
// block's sums over all groups and then applies them to theta (read once,
// written once). Two regions of 64 KB each hold a pair of groups (one per
// half): while the lanes look up groups 2p and 2p+1 in one region, they copy
// the next pair's tables into the other; one barrier per pair separates the
// two. The sums live in tensor memory (TMEM) between pairs, so the chunk is
// not limited by registers: per pair, each 64 KB table copy and its barrier
// serve 4096 blocks. With one or two groups (update_lut8_small_kernel) the
// first region holds them for the whole launch and there is no chunking.
#include <type_traits>

#include "zo_device.cuh"
#include "zo_launch.h"

namespace zo {

constexpr uint32_t kLut8Region = 65536;   // 256 rows x 256 bytes: the tables of two groups
constexpr int kLut8MaxGroups = 48;        // larger K takes update_kernel

// Shared-memory request: two 64 KB regions starting on a 64 KB boundary of
// the shared window, plus the coefficients, 4-probe tables and the chunk's
// virtual blocks (lut8_side_bytes: at most 24 KB), placed in the slack below
// the first region when they fit there (the window starts a few bytes in),
// else after the second: 192 KB covers both cases.
size_t lut8_smem_bytes(int) { return 3 * static_cast<size_t>(kLut8Region) + 16u; }

__device__ __forceinline__ float lds_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}

__device__ __forceinline__ void sts_f32x4(uint32_t addr, float v) {
  asm volatile("st.shared.v4.f32 [%0], {%1, %1, %1, %1};" ::"r"(addr), "f"(v) : "memory");
}

// One 4-probe partial ((s0 a0 + s1 a1) + s2 a2) + s3 a3 for sign nibble i.
__device__ __forceinline__ float quad_partial(const float* a, uint32_t i) {
  float s = (i & 1u) ? a[0] : -a[0];
  s = __fadd_rn(s, (i & 2u) ? a[1] : -a[1]);
  s = __fadd_rn(s, (i & 4u) ? a[2] : -a[2]);
  s = __fadd_rn(s, (i & 8u) ? a[3] : -a[3]);
  return s;
}

// Copy the tables of groups q (and q + 1 when `two`) into the two halves of a
// region. Each thread owns the same 16-byte pieces (four lane copies) of 2048 /
// THREADS rows in every table: row n = p * THREADS / 8 + tid / 8, piece tid mod
// 8, so eight consecutive threads fill one half row (each quarter-warp store
// covers 128 contiguous bytes) and every address is a per-thread base plus a
// constant. All loads are issued before the first store.
//   src_t  shared address of t8 + 4 * (tid / 8)
//   dst_t  region + 256 * (tid / 8) + 16 * (tid mod 8)
template <int THREADS>
__device__ __forceinline__ void lut8_replicate(uint32_t src_t, uint32_t dst_t, int q, bool two) {
  constexpr int S = 2048 / THREADS;                // rows per thread and table
  constexpr uint32_t kRowStep = THREADS / 8;       // rows between a thread's pieces
  float v0[S], v1[S];
  const uint32_t s0 = src_t + static_cast<uint32_t>(q) * 1024u;
#pragma unroll
  for (int p = 0; p < S; ++p) v0[p] = lds_f32(s0 + p * kRowStep * 4u);
  if (two) {
#pragma unroll
    for (int p = 0; p < S; ++p) v1[p] = lds_f32(s0 + 1024u + p * kRowStep * 4u);
  }
#pragma unroll
  for (int p = 0; p < S; ++p) sts_f32x4(dst_t + p * kRowStep * 256u, v0[p]);
  if (two) {
#pragma unroll
    for (int p = 0; p < S; ++p) sts_f32x4(dst_t + 128u + p * kRowStep * 256u, v1[p]);
  }
}

// Add group q's partial of the 16 elements of a block (Philox output x) to acc,
// two elements per packed add. frame: the region's upper half-word, 128 h + 4 l
// in the low byte.
__device__ __forceinline__ void lut8_lookup(float (&acc)[16], const uint4& x, uint32_t frame) {
#pragma unroll
  for (int m = 0; m < 4; ++m) {
    const uint32_t w = word_of(x, m);
#pragma unroll
    for (int j = 0; j < 4; j += 2) {
      // bytes: frame.b0 (lane offset), w.b_j (sign byte -> row), frame.b2, frame.b3 (region)
      const uint32_t a0 = __byte_perm(w, frame, 0x7604u | (static_cast<uint32_t>(j) << 4));
      const uint32_t a1 = __byte_perm(w, frame, 0x7604u | (static_cast<uint32_t>(j + 1) << 4));
      fadd2_rn(acc[4 * m + j], acc[4 * m + j + 1], lds_f32(a0), lds_f32(a1));
    }
  }
}

// A thread's block of the current chunk.
struct Lut8Block {
  int64_t b;       // virtual block (Philox counter)
  int64_t e0;      // first element inside its tensor
  void* base;      // tensor base pointer
  int cnt;         // elements of the block (1..16)
  uint8_t fl;      // tensor flags
  bool act;        // a block this kernel updates
  bool vec16;      // full 32-byte aligned block of a 16-bit tensor (theta already in v)
};

template <uint8_t DT>
__device__ __forceinline__ void lut8_apply16(uint32_t (&v)[8], const float (&acc)[16], const uint4& xp,
                                             const UpdateParams& P, bool do_sum) {
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    if (P.has_pre) v[r] = pre_regs16<DT>(v[r], xp, r, P.pre);
    if (do_sum) {
      const float2 f = unpack2<DT>(v[r]);
      v[r] = pack2<DT>(__fadd_rn(f.x, acc[2 * r]), __fadd_rn(f.y, acc[2 * r + 1]));
    }
  }
}

// Apply the leading perturbation (if any) and the probe sums to a block that
// is not a full, aligned 16-bit one: fp32 blocks and partial last blocks.
__device__ __forceinline__ void lut8_apply_other(const Lut8Block& k, const float (&acc)[16], const UpdateParams& P,
                                              bool do_sum) {
  uint4 xp = make_uint4(0u, 0u, 0u, 0u);
  if (P.has_pre) xp = block_bits(k.b, P.pre.ctr2, P.keys);
  const uint8_t dt = k.fl & kDtypeMask;
  if (dt == kF32 && k.cnt == 16 && (k.fl & kVec32)) {
    float* p = static_cast<float*>(k.base) + k.e0;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      uint32_t v[8];
      ld256(p + 8 * half, v);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        float th = __uint_as_float(v[r]);
        if (P.has_pre) th = add_signed(th, xp, 8 * half + r, P.pre);
        if (do_sum) th = __fadd_rn(th, acc[8 * half + r]);
        v[r] = __float_as_uint(th);
      }
      st256(p + 8 * half, v);
    }
    return;
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    if (i < k.cnt) {
      float th = load_elem(k.base, dt, k.e0 + i);
      if (P.has_pre) th = round_to_storage(dt, add_signed(th, xp, i, P.pre));
      if (do_sum) th = __fadd_rn(th, acc[i]);
      store_elem(k.base, dt, k.e0 + i, th);
    }
  }
}

// Tensor-memory accumulators. A thread's sums for the blocks of its chunk live
// in TMEM between probe-group pairs: 512 threads (16 warps), warp w reaching
// TMEM lanes 32 (w mod 4) .. +31 and, of their 512 columns, the 128 from
// 128 (w / 4); a thread's block j takes 16 columns (one per element). So a CTA
// owns BPT = 8 blocks per thread (4096 blocks, 64 K elements) while its
// registers hold one block's sums at a time, and each table copy and barrier
// serves four times the elements of a register-only chunk of two blocks per
// thread. The copies are what the chunk size is for: a pair's replicated
// tables are 64 KB of shared-memory stores, against 128 KB of lookups per
// 1024 blocks.
constexpr int kLut8Threads = 512;
constexpr uint32_t kTmemCols = 512;

__device__ __forceinline__ void tm_ld16(float (&r)[16], uint32_t taddr) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=f"(r[0]), "=f"(r[1]), "=f"(r[2]), "=f"(r[3]), "=f"(r[4]), "=f"(r[5]), "=f"(r[6]), "=f"(r[7]), "=f"(r[8]),
        "=f"(r[9]), "=f"(r[10]), "=f"(r[11]), "=f"(r[12]), "=f"(r[13]), "=f"(r[14]), "=f"(r[15])
      : "r"(taddr));
}

// Wait for this thread's TMEM loads; the loaded registers pass through the
// wait so that no use of them can be scheduled before it.
__device__ __forceinline__ void tm_wait_ld(float (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+f"(r[0]), "+f"(r[1]), "+f"(r[2]), "+f"(r[3]), "+f"(r[4]), "+f"(r[5]), "+f"(r[6]), "+f"(r[7]),
                 "+f"(r[8]), "+f"(r[9]), "+f"(r[10]), "+f"(r[11]), "+f"(r[12]), "+f"(r[13]), "+f"(r[14]), "+f"(r[15])
               :
               : "memory");
}

__device__ __forceinline__ void tm_st16(uint32_t taddr, const float (&a)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16};" ::"r"(taddr),
      "f"(a[0]), "f"(a[1]), "f"(a[2]), "f"(a[3]), "f"(a[4]), "f"(a[5]), "f"(a[6]), "f"(a[7]), "f"(a[8]), "f"(a[9]),
      "f"(a[10]), "f"(a[11]), "f"(a[12]), "f"(a[13]), "f"(a[14]), "f"(a[15])
      : "memory");
}

__device__ __forceinline__ void tm_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tm_get16(float (&a)[16], uint32_t taddr) {
  tm_ld16(a, taddr);
  tm_wait_ld(a);
}

__device__ __forceinline__ void zero16(float (&a)[16]) {
#pragma unroll
  for (int i = 0; i < 16; ++i) a[i] = 0.0f;
}

// Copy the tables of groups q (and q + 1 when `two`) into the two halves of a
// region, forming each entry T8[n] = T_lo[n & 15] + T_hi[n >> 4] from the
// group's 16-entry 4-probe tables (t4: T_lo then T_hi, 32 floats per group).
// Rows and pieces as in lut8_replicate; a thread's rows are 64 apart, so
// n & 15 is the same in all of them.
template <int THREADS>
__device__ __forceinline__ void lut8_replicate4(uint32_t t4, uint32_t dst_t, int q, bool two) {
  constexpr int S = 2048 / THREADS;
  constexpr uint32_t kRowStep = THREADS / 8;
  static_assert(kRowStep % 16 == 0, "rows of a thread must share n mod 16");
  const uint32_t r0 = threadIdx.x >> 3;
  float v0[S], v1[S];
  const uint32_t g0 = t4 + 128u * static_cast<uint32_t>(q);
  {
    const float lo = lds_f32(g0 + 4u * (r0 & 15u));
#pragma unroll
    for (int p = 0; p < S; ++p) v0[p] = __fadd_rn(lo, lds_f32(g0 + 64u + 4u * ((p * kRowStep + r0) >> 4)));
  }
  if (two) {
    const float lo = lds_f32(g0 + 128u + 4u * (r0 & 15u));
#pragma unroll
    for (int p = 0; p < S; ++p) v1[p] = __fadd_rn(lo, lds_f32(g0 + 192u + 4u * ((p * kRowStep + r0) >> 4)));
  }
#pragma unroll
  for (int p = 0; p < S; ++p) sts_f32x4(dst_t + p * kRowStep * 256u, v0[p]);
  if (two) {
#pragma unroll
    for (int p = 0; p < S; ++p) sts_f32x4(dst_t + 128u + p * kRowStep * 256u, v1[p]);
  }
}

// A thread's tensor while its blocks stay inside it: the table is read again
// only when a block leaves it.
struct Lut8Cursor {
  int t;
  uint32_t tb, te;  // first and one-past-last launch block
  int64_t numel;
  void* base;
  int64_t vbase;    // virtual block of launch block bl of this tensor, minus bl
  uint8_t fl;
};

__device__ __forceinline__ void lut8_seek(const TensorTable& tab, Lut8Cursor& c, uint32_t bl) {
  c.t = advance_tensor(tab, c.t, bl);
  c.tb = tensor_blk_begin(tab, c.t);
  c.te = tab.blk_end[c.t];
  c.numel = tab.numel[c.t];
  c.base = reinterpret_cast<void*>(tab.ptr[c.t]);
  c.vbase = tab.blk_base - static_cast<int64_t>(tab.vdelta[c.t]);
  c.fl = tab.flags[c.t];
}

// Block bl of the launch (bl only grows for a cursor): its tensor and place.
__device__ __forceinline__ void lut8_block_info(const TensorTable& tab, Lut8Cursor& c, uint32_t bl, Lut8Block& k) {
  k.act = bl < tab.blk_total;
  k.vec16 = false;
  if (!k.act) return;
  if (bl >= c.te) lut8_seek(tab, c, bl);
  k.fl = c.fl;
  k.act = !(c.fl & kShift) && bl >= c.tb;
  k.b = c.vbase + static_cast<int64_t>(bl);
  k.e0 = static_cast<int64_t>(bl - c.tb) * 16;
  k.cnt = static_cast<int>(min(static_cast<int64_t>(16), c.numel - k.e0));
  k.base = c.base;
  k.vec16 = k.act && k.cnt == 16 && (c.fl & kVec32) && (c.fl & kDtypeMask) != kF32;
}

// Philox4x32-10 with rounds 0 and 1 split by what they depend on, for a
// launch whose virtual blocks share the counter's high word bhi (every launch
// below 2^36 weights). The counter is (b_lo, bhi, q, 0). Round 0 multiplies
// b_lo (per block) and q (per group); round 1 multiplies the word that came
// from q and bhi (per group) and the one that came from b_lo (per block), so
// both rounds' products are computed once per group (GroupRound01, shared by
// every block) and once per block (BlockRound01, shared by the pair's two
// groups); only their xors and rounds 2-9 are per (block, group). The output
// equals philox10(b_lo, bhi, q, 0) bit for bit.
struct GroupRound01 {
  uint32_t x0;    // lo(M1 q) ^ k0[1]
  uint32_t x2;    // hi(M0 u) ^ k1[1], u = hi(M1 q) ^ bhi ^ k0[0]
  uint32_t lpa1;  // lo(M0 u)
};
struct BlockRound01 {
  uint32_t lpa0;  // lo(M0 b_lo)
  uint32_t hpb1;  // hi(M1 v), v = hi(M0 b_lo) ^ k1[0]
  uint32_t lpb1;  // lo(M1 v)
};
__device__ __forceinline__ GroupRound01 group_round01(uint32_t q, uint32_t bhi, const RoundKeys& rk) {
  const uint64_t pb0 = static_cast<uint64_t>(kPhiloxM1) * q;
  const uint32_t u = static_cast<uint32_t>(pb0 >> 32) ^ bhi ^ rk.k0[0];
  const uint64_t pa1 = static_cast<uint64_t>(kPhiloxM0) * u;
  GroupRound01 g;
  g.x0 = static_cast<uint32_t>(pb0) ^ rk.k0[1];
  g.x2 = static_cast<uint32_t>(pa1 >> 32) ^ rk.k1[1];
  g.lpa1 = static_cast<uint32_t>(pa1);
  return g;
}
__device__ __forceinline__ BlockRound01 block_round01(uint32_t blo, const RoundKeys& rk) {
  const uint64_t pa0 = static_cast<uint64_t>(kPhiloxM0) * blo;
  const uint32_t v = static_cast<uint32_t>(pa0 >> 32) ^ rk.k1[0];
  const uint64_t pb1 = static_cast<uint64_t>(kPhiloxM1) * v;
  BlockRound01 k;
  k.lpa0 = static_cast<uint32_t>(pa0);
  k.hpb1 = static_cast<uint32_t>(pb1 >> 32);
  k.lpb1 = static_cast<uint32_t>(pb1);
  return k;
}
__device__ __forceinline__ uint4 philox_split(const BlockRound01& k, const GroupRound01& g, const RoundKeys& rk) {
  uint32_t c0 = k.hpb1 ^ g.x0, c1 = k.lpb1, c2 = g.x2 ^ k.lpa0, c3 = g.lpa1;
#pragma unroll
  for (int r = 2; r < 10; ++r) philox_round(c0, c1, c2, c3, rk.k0[r], rk.k1[r]);
  return make_uint4(c0, c1, c2, c3);
}

// One step of a probe-group pair: one block of this thread (its sums at TMEM
// address ta) over group q and, when `two`, q + 1, the groups added in order.
// Every lane takes part (an inactive lane's sums are never applied), so the
// step has no per-lane branch; the group-q Philox call runs while the sums
// come in from TMEM.
template <bool FIRST>
__device__ __forceinline__ void lut8_tm_step(uint32_t ta, int64_t b, uint32_t q, bool two, uint32_t frame,
                                             const RoundKeys& keys) {
  float acc[16];
  if (FIRST)
    zero16(acc);
  else
    tm_ld16(acc, ta);
  const uint4 x0 = block_bits(b, q, keys);
  if (!FIRST) tm_wait_ld(acc);
  lut8_lookup(acc, x0, frame);
  if (two) lut8_lookup(acc, block_bits(b, q + 1u, keys), frame | 128u);
  tm_st16(ta, acc);
}

// The same step for a launch whose blocks share the counter's high word:
// blo is the block's low word, g0 / g1 the groups' round-0/1 parts.
template <bool FIRST>
__device__ __forceinline__ void lut8_tm_step_split(uint32_t ta, uint32_t blo, const GroupRound01& g0,
                                                   const GroupRound01& g1, bool two, uint32_t frame,
                                                   const RoundKeys& keys) {
  float acc[16];
  if (FIRST)
    zero16(acc);
  else
    tm_ld16(acc, ta);
  const BlockRound01 k = block_round01(blo, keys);
  const uint4 x0 = philox_split(k, g0, keys);
  if (!FIRST) tm_wait_ld(acc);
  lut8_lookup(acc, x0, frame);
  if (two) lut8_lookup(acc, philox_split(k, g1, keys), frame | 128u);
  tm_st16(ta, acc);
}

// Shared memory besides the two regions: coefficients (8 per group), 4-probe
// tables (32 per group) and the chunk's virtual blocks (one per thread and
// block), below the first region when they fit there, else after the second.
__host__ __device__ constexpr uint32_t lut8_side_bytes(int groups, int bpt) {
  return 160u * static_cast<uint32_t>(groups) + 4u * kLut8Threads * static_cast<uint32_t>(bpt);
}
// Placed after the second region only when the slack below the first is
// smaller than it, so the layout ends within 2 * side + 128 KB of the window's
// start: inside the 192 KB request while side <= 32 KB.
static_assert(lut8_side_bytes(kLut8MaxGroups, 8) <= kLut8Region / 2, "side data must fit the request");

// HIU: every virtual block of the launch has the same counter high word (any
// launch below 2^36 weights), so the steps use the split Philox and a 32-bit
// block word (OPT-30B-shaped set, K = 256: 245.3 -> 235.9 ms, same bits).
template <int BPT, bool HIU>
__global__ void __launch_bounds__(kLut8Threads, 1) update_lut8_kernel(const __grid_constant__ UpdateParams P) {
  constexpr int THREADS = kLut8Threads;
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int skip_s;
  __shared__ uint32_t tmem_s;
  const int G = P.groups;
  const int NP = (G + 1) / 2;  // group pairs: groups 2p, 2p + 1 share one region
  const uint32_t sbase = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  const uint32_t region0 = (sbase + kLut8Region - 1u) & ~(kLut8Region - 1u);
  const uint32_t side = lut8_side_bytes(G, BPT);
  const uint32_t hdr = region0 - sbase >= side ? sbase : region0 + 2u * kLut8Region;
  float* a_s = reinterpret_cast<float*>(smem + (hdr - sbase));  // 8 G coefficients
  float* t4 = a_s + 8 * G;                                      // 32 G 4-probe partials
  uint32_t* vr_s = reinterpret_cast<uint32_t*>(t4 + 32 * G);     // BPT x THREADS virtual blocks

  if (threadIdx.x == 0) skip_s = (P.status != nullptr && *P.status != 0);
  for (int k = threadIdx.x; k < 8 * G; k += THREADS)
    a_s[k] = k < P.K ? __double2float_rn(P.coef_mul * P.coef[k]) : 0.0f;
  __syncthreads();
  const bool skip = skip_s != 0;
  if (skip && !P.has_pre) return;
  const bool do_sum = !skip;  // a failed preconditioner still gets the leading perturbation
  const uint32_t warp = threadIdx.x >> 5;
  const uint32_t t4_s = hdr + 32u * G;
  const uint32_t dst_t = 256u * (threadIdx.x >> 3) + 16u * (threadIdx.x & 7u);
  uint32_t trow = 0;
  if (do_sum) {
    for (int e = threadIdx.x; e < 32 * G; e += THREADS) {
      const float* a = a_s + 8 * (e >> 5) + ((e & 16) ? 4 : 0);
      t4[e] = quad_partial(a, static_cast<uint32_t>(e) & 15u);
    }
    __syncthreads();
    lut8_replicate4<THREADS>(t4_s, region0 + dst_t, 0, G > 1);
    if (warp == 0) {
      __syncwarp();
      const uint32_t dst = static_cast<uint32_t>(__cvta_generic_to_shared(&tmem_s));
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst), "r"(kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tm_fence_before();
    __syncthreads();
    tm_fence_after();
    // TMEM lane 32 (warp mod 4) + lane id, columns from 128 (warp / 4)
    trow = tmem_s + (((warp & 3u) * 32u) << 16) + (warp >> 2) * 128u;
  }

  const TensorTable& tab = P.tab;
  const uint32_t lane = threadIdx.x & 31u;
  constexpr uint32_t chunk = static_cast<uint32_t>(THREADS * BPT);
  const uint32_t per_round = gridDim.x * chunk;
  const uint32_t rounds = (tab.blk_total + per_round - 1u) / per_round;
  uint32_t cur = 0;  // region holding the current pair (0 or 1)
  Lut8Cursor cur0;   // tensor cursor at this thread's first block of the chunk
  cur0.t = 0;
  cur0.te = 0;       // nothing cached yet: the first block seeks

  for (uint32_t rnd = 0; rnd < rounds; ++rnd) {
    // this thread's blocks of the chunk: cb, cb + THREADS, ..
    const uint32_t cb = (rnd * gridDim.x + blockIdx.x) * chunk + threadIdx.x;
    if (do_sum) {
      uint32_t wact = 0;  // blocks of the chunk that some lane of the warp sums
      Lut8Cursor c = cur0;
#pragma unroll
      for (int j = 0; j < BPT; ++j) {
        Lut8Block k;
        lut8_block_info(tab, c, cb + static_cast<uint32_t>(j * THREADS), k);
        // HIU: the virtual block's low word; otherwise its offset from blk_base
        vr_s[j * THREADS + threadIdx.x] =
            k.act ? static_cast<uint32_t>(HIU ? static_cast<uint64_t>(k.b) : static_cast<uint64_t>(k.b - tab.blk_base))
                  : 0u;
        if (__any_sync(0xFFFFFFFFu, k.act)) wact |= 1u << j;
        // theta is read after all pairs: bring it into L2 meanwhile
        if (k.vec16) asm volatile("prefetch.L2 [%0];" ::"l"(static_cast<uint16_t*>(k.base) + k.e0));
      }
      for (int pr = 0; pr < NP; ++pr) {
        const uint32_t frame = ((region0 + cur * kLut8Region) & 0xFFFF0000u) | (lane << 2);
        const uint32_t q = 2u * static_cast<uint32_t>(pr);
        const bool two = static_cast<int>(q) + 1 < G;
        const auto run = [&](auto first) {
          if constexpr (HIU) {
            const uint32_t bhi = static_cast<uint32_t>(static_cast<uint64_t>(tab.blk_base) >> 32);
            const GroupRound01 g0 = group_round01(q, bhi, P.keys);
            const GroupRound01 g1 = group_round01(q + 1u, bhi, P.keys);
#pragma unroll
            for (int j = 0; j < BPT; ++j) {
              if (!((wact >> j) & 1u)) continue;  // no lane of the warp has this block
              const uint32_t blo = vr_s[j * THREADS + threadIdx.x];
              lut8_tm_step_split<decltype(first)::value>(trow + 16u * static_cast<uint32_t>(j), blo, g0, g1, two,
                                                         frame, P.keys);
            }
          } else {
#pragma unroll
            for (int j = 0; j < BPT; ++j) {
              if (!((wact >> j) & 1u)) continue;  // no lane of the warp has this block
              const int64_t b = tab.blk_base + vr_s[j * THREADS + threadIdx.x];
              lut8_tm_step<decltype(first)::value>(trow + 16u * static_cast<uint32_t>(j), b, q, two, frame, P.keys);
            }
          }
        };
        if (pr == 0)
          run(std::true_type());
        else
          run(std::false_type());
        tm_wait_st();  // this pair's sums are in TMEM before the next pair reads them
        if (NP > 1) {
          // the next pair (wrapping to pair 0 for the next chunk) into the other region
          const int qn = pr + 1 < NP ? static_cast<int>(q) + 2 : 0;
          lut8_replicate4<THREADS>(t4_s, region0 + (cur ^ 1u) * kLut8Region + dst_t, qn, qn + 1 < G);
          __syncthreads();
          cur ^= 1u;
        }
      }
    }
    // Apply: each block's sums read back from TMEM and added to theta (in L2
    // by now). Full aligned 16-bit blocks here; the rare others (fp32, partial
    // last blocks) in a loop of their own, which keeps their code out of this one.
    Lut8Cursor c = cur0;
    bool others = false;
#pragma unroll 1
    for (int j = 0; j < BPT; ++j) {
      Lut8Block k;
      lut8_block_info(tab, c, cb + static_cast<uint32_t>(j * THREADS), k);
      others |= k.act && !k.vec16;
      uint32_t v[8];
      if (k.vec16) ld256(static_cast<uint16_t*>(k.base) + k.e0, v);
      float acc[16];
      zero16(acc);
      if (do_sum && __any_sync(0xFFFFFFFFu, k.vec16)) tm_get16(acc, trow + 16u * static_cast<uint32_t>(j));
      if (k.vec16) {
        uint4 xp = make_uint4(0u, 0u, 0u, 0u);
        if (P.has_pre) xp = block_bits(k.b, P.pre.ctr2, P.keys);
        if ((k.fl & kDtypeMask) == kBF16)
          lut8_apply16<kBF16>(v, acc, xp, P, do_sum);
        else
          lut8_apply16<kF16>(v, acc, xp, P, do_sum);
        st256(static_cast<uint16_t*>(k.base) + k.e0, v);
      }
    }
    if (__any_sync(0xFFFFFFFFu, others)) {
      Lut8Cursor c2 = cur0;
#pragma unroll 1
      for (int j = 0; j < BPT; ++j) {
        Lut8Block k;
        lut8_block_info(tab, c2, cb + static_cast<uint32_t>(j * THREADS), k);
        const bool mine = k.act && !k.vec16;
        float acc[16];
        zero16(acc);
        if (do_sum && __any_sync(0xFFFFFFFFu, mine)) tm_get16(acc, trow + 16u * static_cast<uint32_t>(j));
        if (mine) lut8_apply_other(k, acc, P, do_sum);
      }
    }
    cur0 = c;
  }
  if (do_sum) {
    tm_fence_before();
    __syncthreads();
    tm_fence_after();
    if (warp == 0) {
      __syncwarp();
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_s), "r"(kTmemCols) : "memory");
    }
  }
}

// ---------------------------------------------------------------------------
// One or two probe groups (K <= 16): both tables stay in the first region for
// the whole launch, so there is no chunking and no barrier. The kernel walks
// blocks grid-stride like the perturbation passes, the next block's 256-bit
// load issued before the current block is computed, and every element takes
// its one or two lookups and is stored at once: the same sums, in the same
// order (0 + T8_0 [+ T8_1]), as the chunked kernel. The leading perturbation
// reuses the Philox word of its own group when it is one of the two. The group
// count and the leading perturbation's case are template arguments: with
// 64 registers a thread (1024 threads), the run-time flags cost 7-14 % of
// the time of this issue-bound loop.
// ---------------------------------------------------------------------------
constexpr int kSmallThreads = 1024;
size_t lut8_small_smem_bytes() { return 2 * static_cast<size_t>(kLut8Region) + 16u; }

struct SmallCursor {
  int t;
  uint32_t tb, te, n16;  // first and one-past-last launch block; full aligned 16-bit blocks from tb
  uint32_t vd;           // launch block minus virtual block offset
  uint16_t* tp;
  uint8_t dt;
};

__device__ __forceinline__ void small_seek(const TensorTable& tab, SmallCursor& c, uint32_t b) {
  c.t = advance_tensor(tab, c.t, b);
  c.tb = tensor_blk_begin(tab, c.t);
  c.te = tab.blk_end[c.t];
  const uint8_t fl = tab.flags[c.t];
  c.dt = fl & kDtypeMask;
  c.n16 = ((fl & kVec32) && c.dt != kF32) ? static_cast<uint32_t>(tab.numel[c.t] / 16) : 0u;
  c.vd = tab.vdelta[c.t];
  c.tp = reinterpret_cast<uint16_t*>(tab.ptr[c.t]);
}

// Sums of elements e and e + 1 (e even) of a block, 0 + T8_0 [+ T8_1] each,
// from the Philox words of groups 0 and 1, two elements per packed add.
template <int E>
__device__ __forceinline__ float2 small_sum2(const uint4& x0, const uint4& x1, uint32_t frame, bool two) {
  constexpr uint32_t sel0 = 0x7604u | (static_cast<uint32_t>(E & 3) << 4);
  constexpr uint32_t sel1 = 0x7604u | (static_cast<uint32_t>((E + 1) & 3) << 4);
  float lo = 0.0f, hi = 0.0f;
  const uint32_t w0 = word_of(x0, E >> 2);
  fadd2_rn(lo, hi, lds_f32(__byte_perm(w0, frame, sel0)), lds_f32(__byte_perm(w0, frame, sel1)));
  if (two) {
    const uint32_t w1 = word_of(x1, E >> 2);
    fadd2_rn(lo, hi, lds_f32(__byte_perm(w1, frame | 128u, sel0)), lds_f32(__byte_perm(w1, frame | 128u, sel1)));
  }
  return make_float2(lo, hi);
}

// theta pair + the leading perturbation's signed scales, one packed add.
__device__ __forceinline__ void add_signed2(float2& f, const uint4& x, int i, const PerturbOp& op) {
  // the probe bit moved to bit 31 by a multiply (PerturbOp::mul): the
  // multiply-add pipe instead of the integer ALU, the busier one here
  fadd2_rn(f.x, f.y, __uint_as_float(op.nscale_bits ^ ((word_of(x, i >> 2) * op.mul[i & 3]) & 0x80000000u)),
           __uint_as_float(op.nscale_bits ^ ((word_of(x, (i + 1) >> 2) * op.mul[(i + 1) & 3]) & 0x80000000u)));
}

template <uint8_t DT, bool TWO>
__device__ __forceinline__ void small_block16(uint32_t (&v)[8], const uint4& x0, const uint4& x1, const uint4& xp,
                                              uint32_t frame, bool pre, const UpdateParams& P, bool do_sum) {
  constexpr bool two = TWO;
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    float2 f = unpack2<DT>(v[r]);
    if (pre) {
      add_signed2(f, xp, 2 * r, P.pre);
      v[r] = pack2<DT>(f.x, f.y);  // the perturbed value is rounded to storage first
      f = unpack2<DT>(v[r]);
    }
    if (do_sum) {
      float2 acc;
      switch (r) {  // element indices must be constants for the word and byte selects
        case 0: acc = small_sum2<0>(x0, x1, frame, two); break;
        case 1: acc = small_sum2<2>(x0, x1, frame, two); break;
        case 2: acc = small_sum2<4>(x0, x1, frame, two); break;
        case 3: acc = small_sum2<6>(x0, x1, frame, two); break;
        case 4: acc = small_sum2<8>(x0, x1, frame, two); break;
        case 5: acc = small_sum2<10>(x0, x1, frame, two); break;
        case 6: acc = small_sum2<12>(x0, x1, frame, two); break;
        default: acc = small_sum2<14>(x0, x1, frame, two); break;
      }
      fadd2_rn(f.x, f.y, acc.x, acc.y);
      v[r] = pack2<DT>(f.x, f.y);
    }
  }
}

// Any other block of the launch: fp32, a partial last block, padding, or an
// unaligned tensor (update_shift_kernel's).
template <int TAG>
__device__ __noinline__ void small_block_other(const TensorTable& tab, int t, uint32_t b, const UpdateParams& P,
                                               uint32_t frame, bool do_sum) {
  const uint32_t tb = tensor_blk_begin(tab, t);
  const uint8_t fl = tab.flags[t];
  if ((fl & kShift) || b < tb) return;
  Lut8Block k;
  k.b = virtual_block(tab, t, b);
  k.e0 = static_cast<int64_t>(b - tb) * 16;
  k.cnt = static_cast<int>(min(static_cast<int64_t>(16), tab.numel[t] - k.e0));
  k.base = reinterpret_cast<void*>(tab.ptr[t]);
  k.fl = fl;
  k.act = true;
  k.vec16 = false;
  float acc[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) acc[i] = 0.0f;
  if (do_sum) {
    lut8_lookup(acc, block_bits(k.b, 0u, P.keys), frame);
    if (P.groups > 1) lut8_lookup(acc, block_bits(k.b, 1u, P.keys), frame | 128u);
  }
  lut8_apply_other(k, acc, P, do_sum);
}

// Leading perturbation of the small kernel's instantiations: on a Philox word
// the sums also use (group 0 or 1), on its own word, or decided at run time
// (no leading perturbation, or any).
constexpr int kPreShared = 1, kPreOwn = 2, kPreRuntime = 3;

template <int PRE, bool TWO>
__global__ void __launch_bounds__(kSmallThreads, 1) update_lut8_small_kernel(const __grid_constant__ UpdateParams P) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int skip_s;
  const int G = P.groups;  // 1 or 2
  const uint32_t sbase = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  const uint32_t region0 = (sbase + kLut8Region - 1u) & ~(kLut8Region - 1u);
  // coefficients and unreplicated tables (2 KB at most) below the region, or after it when the window starts on
  // a 64 KB boundary
  const uint32_t hdr = region0 - sbase >= 32u * G + 1024u * G ? sbase : region0 + kLut8Region;
  float* a_s = reinterpret_cast<float*>(smem + (hdr - sbase));
  float* t8 = a_s + 8 * G;
  if (threadIdx.x == 0) skip_s = (P.status != nullptr && *P.status != 0);
  for (int k = threadIdx.x; k < 8 * G; k += kSmallThreads)
    a_s[k] = k < P.K ? __double2float_rn(P.coef_mul * P.coef[k]) : 0.0f;
  __syncthreads();
  const bool skip = skip_s != 0;
  const bool has_pre = PRE == kPreRuntime ? P.has_pre : true;
  if (skip && !has_pre) return;
  const bool do_sum = !skip;
  if (do_sum) {
    for (int e = threadIdx.x; e < 256 * G; e += kSmallThreads) {
      const float* a = a_s + 8 * (e >> 8);
      const uint32_t n = static_cast<uint32_t>(e) & 255u;
      t8[e] = __fadd_rn(quad_partial(a, n & 15u), quad_partial(a + 4, n >> 4));
    }
    __syncthreads();
    const uint32_t src_t = hdr + 32u * G + 4u * (threadIdx.x >> 3);
    const uint32_t dst_t = 256u * (threadIdx.x >> 3) + 16u * (threadIdx.x & 7u);
    lut8_replicate<kSmallThreads>(src_t, region0 + dst_t, 0, G > 1);
    __syncthreads();
  }
  const TensorTable& tab = P.tab;
  const uint32_t total = tab.blk_total;
  const uint32_t stride = gridDim.x * kSmallThreads;
  const uint32_t frame = (region0 & 0xFFFF0000u) | ((threadIdx.x & 31u) << 2);
  constexpr bool two = TWO;
  // the leading perturbation's Philox word: group 0's, group 1's, or its own
  // the leading perturbation's Philox word: none (-1), group 0's or group 1's (0, 1), or its own (2)
  const int pre_src = PRE == kPreOwn ? 2
                      : PRE == kPreShared ? (P.pre.ctr2 == 1u ? 1 : 0)
                      : (!P.has_pre ? -1 : (P.pre.ctr2 == 0u ? 0 : (P.pre.ctr2 == 1u && two ? 1 : 2)));
  uint32_t b = blockIdx.x * kSmallThreads + threadIdx.x;
  if (b >= total) return;
  SmallCursor c;
  c.t = 0;
  small_seek(tab, c, b);
  int t = c.t;
  uint8_t dt = c.dt;
  uint32_t vd = c.vd;
  bool fast = b - c.tb < c.n16;
  uint16_t* p = c.tp + static_cast<size_t>(b - c.tb) * 16;
  uint32_t v[8];
  if (fast) ld256(p, v);
  while (true) {
    const uint32_t bn = b + stride;
    bool fastn = false;
    uint16_t* pn = nullptr;
    uint32_t vn[8];
    if (bn < total) {
      if (bn >= c.te) small_seek(tab, c, bn);
      fastn = bn - c.tb < c.n16;
      pn = c.tp + static_cast<size_t>(bn - c.tb) * 16;
      if (fastn) ld256(pn, vn);
    }
    if (fast) {
      const int64_t vb = tab.blk_base + (b - vd);
      uint4 x0 = make_uint4(0u, 0u, 0u, 0u), x1 = x0, xp = x0;
      if (do_sum || pre_src == 0 || pre_src == 1) {
        x0 = block_bits(vb, 0u, P.keys);
        if (two) x1 = block_bits(vb, 1u, P.keys);
      }
      if (pre_src == 0) xp = x0;
      if (pre_src == 1) xp = x1;
      if (pre_src == 2) xp = block_bits(vb, P.pre.ctr2, P.keys);
      if (dt == kBF16)
        small_block16<kBF16, TWO>(v, x0, x1, xp, frame, has_pre, P, do_sum);
      else
        small_block16<kF16, TWO>(v, x0, x1, xp, frame, has_pre, P, do_sum);
      st256(p, v);
    } else {
      small_block_other<2 * PRE + TWO>(tab, t, b, P, frame, do_sum);
    }
    if (bn >= total) break;
    b = bn;
    t = c.t;
    dt = c.dt;
    vd = c.vd;
    fast = fastn;
    p = pn;
#pragma unroll
    for (int r = 0; r < 8; ++r) v[r] = vn[r];
  }
}

template <int BPT>
cudaError_t launch_lut8_cfg(const UpdateParams& p, int grid, cudaStream_t stream) {
  // every virtual block of the launch lies in [blk_base, blk_base + blk_total)
  const uint64_t first = static_cast<uint64_t>(p.tab.blk_base);
  const uint64_t last = first + (p.tab.blk_total > 0 ? p.tab.blk_total - 1u : 0u);
  if ((first >> 32) == (last >> 32))
    update_lut8_kernel<BPT, true><<<grid, kLut8Threads, lut8_smem_bytes(p.groups), stream>>>(p);
  else
    update_lut8_kernel<BPT, false><<<grid, kLut8Threads, lut8_smem_bytes(p.groups), stream>>>(p);
  return cudaGetLastError();
}

template <int BPT>
cudaError_t lut8_prepare_cfg(int groups, int* blocks_per_sm) {
  // the limit covers every group count, so later launches with more groups still fit
  cudaError_t e = cudaFuncSetAttribute(update_lut8_kernel<BPT, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(lut8_smem_bytes(kLut8MaxGroups)));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(update_lut8_kernel<BPT, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(lut8_smem_bytes(kLut8MaxGroups)));
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, update_lut8_kernel<BPT, false>, kLut8Threads,
                                                       lut8_smem_bytes(groups));
}

bool lut8_supported(int groups, int packing) { return packing == kPacking1 && groups >= 1 && groups <= kLut8MaxGroups; }

cudaError_t lut8_prepare(int groups, int* blocks_per_sm) {
  if (groups <= 2) {
    const int lim = static_cast<int>(lut8_small_smem_bytes());
    cudaError_t e = cudaSuccess;
    const void* kernels[] = {
        reinterpret_cast<const void*>(update_lut8_small_kernel<kPreShared, false>),
        reinterpret_cast<const void*>(update_lut8_small_kernel<kPreShared, true>),
        reinterpret_cast<const void*>(update_lut8_small_kernel<kPreOwn, false>),
        reinterpret_cast<const void*>(update_lut8_small_kernel<kPreOwn, true>),
        reinterpret_cast<const void*>(update_lut8_small_kernel<kPreRuntime, false>),
        reinterpret_cast<const void*>(update_lut8_small_kernel<kPreRuntime, true>)};
    for (const void* k : kernels)
      if (e == cudaSuccess) e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, update_lut8_small_kernel<kPreRuntime, true>,
                                                         kSmallThreads, lut8_small_smem_bytes());
  }
  cudaError_t e = lut8_prepare_cfg<2>(groups, blocks_per_sm);
  if (e == cudaSuccess) e = lut8_prepare_cfg<4>(groups, blocks_per_sm);
  if (e == cudaSuccess) e = lut8_prepare_cfg<8>(groups, blocks_per_sm);
  return e;
}

// Blocks per thread: the largest of 8, 4, 2 that still gives every SM a chunk.
int lut8_bpt(uint32_t blk_total, int sms) {
  for (int bpt = 8; bpt > 2; bpt /= 2)
    if (static_cast<int64_t>(blk_total) >= static_cast<int64_t>(sms) * kLut8Threads * bpt) return bpt;
  return 2;
}


cudaError_t launch_update_lut8(const UpdateParams& p, int sms, int blocks_per_sm, cudaStream_t stream) {
  const int64_t total = p.tab.blk_total;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  if (p.groups <= 2) {
    const int64_t want = (total + kSmallThreads - 1) / kSmallThreads;
    const int g = static_cast<int>(want < cap ? want : cap);
    const size_t sm = lut8_small_smem_bytes();
    // with a leading perturbation: its Philox word one of the sums' or its own;
    // without one, the run-time instantiation (faster there: its registers are
    // laid out for the leading perturbation and it does not spill)
    const bool two = p.groups == 2;
    const int pre = !p.has_pre ? kPreRuntime
                               : (p.pre.ctr2 == 0u || (p.pre.ctr2 == 1u && two) ? kPreShared : kPreOwn);
    if (pre == kPreShared && two)
      update_lut8_small_kernel<kPreShared, true><<<g, kSmallThreads, sm, stream>>>(p);
    else if (pre == kPreShared)
      update_lut8_small_kernel<kPreShared, false><<<g, kSmallThreads, sm, stream>>>(p);
    else if (pre == kPreOwn && two)
      update_lut8_small_kernel<kPreOwn, true><<<g, kSmallThreads, sm, stream>>>(p);
    else if (pre == kPreOwn)
      update_lut8_small_kernel<kPreOwn, false><<<g, kSmallThreads, sm, stream>>>(p);
    else if (two)
      update_lut8_small_kernel<kPreRuntime, true><<<g, kSmallThreads, sm, stream>>>(p);
    else
      update_lut8_small_kernel<kPreRuntime, false><<<g, kSmallThreads, sm, stream>>>(p);
    return cudaGetLastError();
  }
  // one CTA per chunk of 512 * BPT blocks, at most the resident CTAs
  const int bpt = lut8_bpt(p.tab.blk_total, sms);
  const int64_t chunk = static_cast<int64_t>(kLut8Threads) * bpt;
  const int64_t want = (total + chunk - 1) / chunk;
  const int grid = static_cast<int>(want < cap ? want : cap);
  switch (bpt) {
    case 8: return launch_lut8_cfg<8>(p, grid, stream);
    case 4: return launch_lut8_cfg<4>(p, grid, stream);
    default: return launch_lut8_cfg<2>(p, grid, stream);
  }
}

}  // namespace zo
