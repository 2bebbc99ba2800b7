// zo_api.cu -- the extern "C" entry points declared in include/zo.h: argument
// validation, Philox key expansion, tensor-table planning and launch sizing.
// Everything here runs on the host and only enqueues kernels.
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <vector>

#include <cuda_runtime.h>

#include "zo.h"
#include "zo_launch.h"

namespace {

using zo::PerturbParams;
using zo::RoundKeys;
using zo::TensorTable;
using zo::UpdateParams;

thread_local char g_last_cuda_error[256] = "";

int cuda_fail(cudaError_t e, const char* where) {
  std::snprintf(g_last_cuda_error, sizeof(g_last_cuda_error), "%s: %s (%s)", where, cudaGetErrorName(e),
                cudaGetErrorString(e));
  return ZO_ERR_CUDA;
}

// Philox4x32 key schedule: round r uses (lo + r * W0, hi + r * W1) mod 2^32.
RoundKeys expand_keys(uint64_t seed) {
  RoundKeys k;
  uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
  for (int r = 0; r < 10; ++r) {
    k.k0[r] = k0;
    k.k1[r] = k1;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return k;
}

int elem_size(int32_t dtype) { return dtype == ZO_F32 ? 4 : 2; }

// Probe packing of every later call (1 or 8 generated bits per weight and probe).
std::atomic<int> g_packing{zo::kPacking1};

// Third Philox counter word and sign bit of probe k under the current packing.
void probe_counter(uint32_t k, int packing, uint32_t* ctr2, uint32_t* bit) {
  if (packing == zo::kPacking8) {
    *ctr2 = k;
    *bit = 0;
  } else {
    *ctr2 = k >> 3;
    *bit = k & 7u;
  }
}

// theta <- rn(theta + scale z_k) as a kernel operand.
zo::PerturbOp make_op(uint32_t k, float scale, int packing) {
  zo::PerturbOp op;
  probe_counter(k, packing, &op.ctr2, &op.bit);
  uint32_t u;
  std::memcpy(&u, &scale, sizeof(u));
  op.nscale_bits = u ^ 0x80000000u;  // -scale: the probe bit flips it to +scale
  for (uint32_t m = 0; m < 4; ++m) op.mul[m] = 1u << (31u - 8u * m - op.bit);
  return op;
}

// Resident perturb blocks per SM. The passes are HBM-bound and each thread
// keeps two 32-byte loads in flight. The single-op pass streams fastest with
// four 256-thread blocks per SM (3 -> 90.6 %, 4 -> 97.7 %, 5 -> 93.0 % of the
// copy bandwidth on the 60 GB OPT-30B-shaped set), the out-of-place pair pass
// with three. The two-op pass has three candidate (loop, blocks per SM)
// configurations, timed on the caller's list (TwoOpTuner below).
constexpr int kPerturbBlocksPerSm = 4;
constexpr int kPairBlocksPerSm = 3;
constexpr int kShiftBlocksPerSm = 4;   // pair_shift_kernel: 256 threads, at most 64 registers
constexpr int kTwoOpCandidates = 3;
constexpr int kTwoOpLoop[kTwoOpCandidates] = {zo::kLoopRuns, zo::kLoopRuns, zo::kLoopBlocks};
constexpr int kTwoOpBlocksPerSm[kTwoOpCandidates] = {3, 4, 4};

// The update is issue-bound; four waves of its blocks per SM keep more warps
// eligible than one persistent wave (measured +3 % at K = 64 and 256).
constexpr int kUpdateWaves = 4;

// Packing-1 updates with up to 48 probe groups take the 8-probe-table kernel
// (update_lut8_kernel); larger K and packing 8 take update_kernel. Measured
// on the OPT-1.3B-shaped bf16 set against update_kernel: K = 8 1.08 vs 1.17
// ms, K = 16 1.34 vs 1.60, K = 64 3.83 vs 4.21, K = 256 12.9 vs 14.7 (same
// bits); on the OPT-30B-shaped fp16 set at K = 256 292 vs 332 ms.
#ifndef ZO_LUT8_MIN_GROUPS
#define ZO_LUT8_MIN_GROUPS 1
#endif
constexpr int kLut8MinGroups = ZO_LUT8_MIN_GROUPS;

// Per-device launch facts, filled once per device.
struct DeviceInfo {
  int sms = 0;
  int perturb_bps = 0;                    // single-op perturb blocks per SM
  int two_op_bps[kTwoOpCandidates] = {};  // two-op perturb blocks per SM, by candidate
  int pair_bps = 0;                       // perturb_pair blocks per SM
  int shift_bps[2][3] = {};               // perturb_shift blocks per SM, by operation count and dtype
  int update_bps[2][zo::kMaxGroups + 1] = {};  // by packing (1, 8) and probe-group count
  int update_shift_bps[2][3][zo::kMaxGroups + 1] = {};  // update_shift_kernel: packing, dtype, group count
  int lut8_bps[zo::kMaxGroups + 1] = {};  // update_lut8_kernel, by group count
};
constexpr int kMaxDevices = 64;
DeviceInfo g_dev[kMaxDevices];
std::mutex g_dev_mu;

int device_info(DeviceInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return ZO_ERR_ARG;
  std::lock_guard<std::mutex> lock(g_dev_mu);
  DeviceInfo& d = g_dev[dev];
  if (d.sms == 0) {
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    int bps = 0;
    e = zo::perturb_blocks_per_sm(1, zo::kLoopBlocks, &bps);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy(perturb)");
    d.perturb_bps = bps < 1 ? 1 : (bps < kPerturbBlocksPerSm ? bps : kPerturbBlocksPerSm);
    for (int i = 0; i < kTwoOpCandidates; ++i) {
      e = zo::perturb_blocks_per_sm(2, kTwoOpLoop[i], &bps);
      if (e != cudaSuccess) return cuda_fail(e, "occupancy(perturb2)");
      d.two_op_bps[i] = bps < 1 ? 1 : (bps < kTwoOpBlocksPerSm[i] ? bps : kTwoOpBlocksPerSm[i]);
    }
    e = zo::pair_blocks_per_sm(&bps);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy(perturb_pair)");
    d.pair_bps = bps < 1 ? 1 : (bps < kPairBlocksPerSm ? bps : kPairBlocksPerSm);
    for (int nops = 1; nops <= 2; ++nops) {
      for (uint8_t dt = 0; dt < 3; ++dt) {
        e = zo::shift_blocks_per_sm(nops, dt, &bps);
        if (e != cudaSuccess) return cuda_fail(e, "occupancy(perturb_shift)");
        d.shift_bps[nops - 1][dt] = bps < 1 ? 1 : bps;
      }
    }
    d.sms = sms;
  }
  *out = &d;
  return ZO_OK;
}

int update_shift_blocks_per_sm(DeviceInfo* d, int groups, int packing, uint8_t dt, int* out) {
  std::lock_guard<std::mutex> lock(g_dev_mu);
  int& slot = d->update_shift_bps[packing == zo::kPacking8 ? 1 : 0][dt][groups];
  if (slot == 0) {
    int bps = 0;
    cudaError_t e = zo::update_shift_blocks_per_sm(groups, packing, dt, &bps);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy(update_shift)");
    slot = bps > 0 ? bps : 1;
  }
  *out = slot;
  return ZO_OK;
}

// Also raises the kernel's dynamic shared-memory limit (once per device and
// group count, before the first launch).
int lut8_blocks_per_sm(DeviceInfo* d, int groups, int* out) {
  std::lock_guard<std::mutex> lock(g_dev_mu);
  int& slot = d->lut8_bps[groups];
  if (slot == 0) {
    int bps = 0;
    cudaError_t e = zo::lut8_prepare(groups, &bps);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy(update_lut8)");
    slot = bps > 0 ? bps : 1;
  }
  *out = slot;
  return ZO_OK;
}

int update_blocks_per_sm(DeviceInfo* d, int groups, int packing, int* out) {
  std::lock_guard<std::mutex> lock(g_dev_mu);
  int& slot = d->update_bps[packing == zo::kPacking8 ? 1 : 0][groups];
  if (slot == 0) {
    int bps = 0;
    cudaError_t e = zo::update_blocks_per_sm(groups, packing, &bps);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy(update)");
    slot = bps > 0 ? bps : 1;
  }
  *out = slot;
  return ZO_OK;
}

// Checks a parameter list; *packing (optional) receives the probe packing
// its tensors ask for (zo_tensor.packing: 0 = the process default, else 1
// or 8, the same for every tensor of the list) resolved to 1 or 8.
int validate_params(const zo_tensor* params, int32_t n, int* packing = nullptr) {
  if (n < 0) return ZO_ERR_ARG;
  if (n > 0 && params == nullptr) return ZO_ERR_ARG;
  int64_t blocks = 0;
  const int32_t pk = n > 0 ? params[0].packing : 0;
  if (pk != 0 && pk != zo::kPacking1 && pk != zo::kPacking8) return ZO_ERR_ARG;
  if (packing != nullptr) *packing = pk != 0 ? pk : g_packing.load();
  for (int32_t t = 0; t < n; ++t) {
    const zo_tensor& p = params[t];
    if (p.numel < 0 || p.packing != pk) return ZO_ERR_ARG;
    if (p.dtype != ZO_F32 && p.dtype != ZO_BF16 && p.dtype != ZO_F16) return ZO_ERR_DTYPE;
    if (p.numel > 0 && p.ptr == nullptr) return ZO_ERR_ARG;
    if (reinterpret_cast<uintptr_t>(p.ptr) % static_cast<uintptr_t>(elem_size(p.dtype)) != 0) return ZO_ERR_ALIGN;
    const int64_t nb = (p.numel + 15) / 16;
    if (nb >= zo::kMaxLaunchBlocks) return ZO_ERR_ARG;          // one tensor must fit one launch
    if (nb > (INT64_C(1) << 58) - blocks) return ZO_ERR_ARG;   // virtual index space
    blocks += nb;
  }
  return ZO_OK;
}

// Fill `tab` with tensors t0, t0+1, ... while the launch holds fewer than
// kMaxTensorsPerLaunch tensors and fewer than kMaxLaunchBlocks launch blocks;
// the launch's first block has virtual index blk_base. In the launch
// numbering every tensor starts on a multiple of kLaunchAlign blocks (see
// TensorTable). Returns the first tensor not taken; *nblocks receives the
// virtual blocks the launch covers (tab.blk_total its launch blocks).
int32_t fill_table(TensorTable& tab, const zo_tensor* params, int32_t t0, int32_t n, int64_t blk_base,
                   int64_t* nblocks) {
  tab.n = 0;
  tab.blk_base = blk_base;
  int64_t b = 0;  // launch blocks so far
  int64_t v = 0;  // virtual blocks so far
  int32_t t = t0;
  for (; t < n && tab.n < zo::kMaxTensorsPerLaunch; ++t) {
    const zo_tensor& p = params[t];
    const int64_t nb = (p.numel + 15) / 16;
    const int64_t start = (b + zo::kLaunchAlign - 1) / zo::kLaunchAlign * zo::kLaunchAlign;
    if (tab.n > 0 && start + nb >= zo::kMaxLaunchBlocks) break;
    const int i = tab.n++;
    tab.vdelta[i] = static_cast<uint32_t>(start - v);
    b = start + nb;
    v += nb;
    tab.blk_end[i] = static_cast<uint32_t>(b);
    tab.ptr[i] = reinterpret_cast<uint64_t>(p.ptr);
    tab.numel[i] = p.numel;
    uint8_t fl = static_cast<uint8_t>(p.dtype);
    if (reinterpret_cast<uintptr_t>(p.ptr) % 32 == 0) fl |= zo::kVec32;
    tab.flags[i] = fl;
  }
  tab.blk_total = static_cast<uint32_t>(b);
  *nblocks = v;
  return t;
}

int grid_for(int64_t blocks, int sms, int bps) {
  const int64_t want = (blocks + zo::kThreads - 1) / zo::kThreads;
  const int64_t cap = static_cast<int64_t>(sms) * bps;
  const int64_t g = want < cap ? want : cap;
  return static_cast<int>(g < 1 ? 1 : g);
}

// Choice of the two-op configuration per parameter list. All candidates give
// the same bits; which is fastest depends on the tensor sizes (measured: runs
// with 3 blocks per SM on the OPT-30B-shaped set, one block per iteration with
// 4 on the Qwen3-8B-shaped one, runs with 4 on the OPT-1.3B-shaped one, the
// spread between candidates from 1 % to 12 %). The first calls on a list
// (keyed by its sizes, dtypes, alignments and device, and by whether the two
// probes fall in one group of 8 or in two) run the candidates in turn, three
// rounds each (one for the two-group calls), each call between two events on
// the caller's stream; once all those events have completed (polled, never
// waited for), later calls use the candidate with the shortest time (the
// shortest of its rounds). Calls made while the stream is being captured
// into a graph, or before a decision, use candidate 0.
// After a failed runtime call of this file's own bookkeeping (events, capture
// query): reset the thread's last error only when it is that call's error, so
// an unrelated error the caller has not collected yet stays pending.
void clear_own_error(cudaError_t e) {
  if (e != cudaSuccess && cudaPeekAtLastError() == e) cudaGetLastError();
}

class TwoOpTuner {
 public:
  // Candidate for this call; *slot receives the trial index when the call's
  // launches must be bracketed by that trial's events, else -1.
  int pick(uint64_t key, int rounds, cudaStream_t s, int* slot) {
    *slot = -1;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    const cudaError_t ce = cudaStreamIsCapturing(s, &cap);
    if (ce != cudaSuccess || cap != cudaStreamCaptureStatusNone) {
      clear_own_error(ce);
      return 0;
    }
    std::lock_guard<std::mutex> lock(mu_);
    Entry* e = find(key, rounds);
    if (e == nullptr) return 0;
    if (e->chosen >= 0) return e->chosen;
    decide(*e);
    if (e->chosen >= 0) return e->chosen;
    if (e->next < e->trials) {
      *slot = e->next++;
      return *slot % kTwoOpCandidates;
    }
    return 0;
  }

  void record(uint64_t key, int slot, int which, cudaStream_t s) {
    std::lock_guard<std::mutex> lock(mu_);
    Entry* e = find(key, 0);
    if (e == nullptr || e->ev[slot][which] == nullptr) return;
    const cudaError_t er = cudaEventRecord(e->ev[slot][which], s);
    if (er != cudaSuccess) {
      clear_own_error(er);
      e->failed = true;
    }
  }

 private:
  static constexpr int kMaxRounds = 3;
  static constexpr int kTrials = kMaxRounds * kTwoOpCandidates;

  struct Entry {
    uint64_t key = 0;
    int chosen = -1;
    int next = 0;  // next trial; trial i runs candidate i % kTwoOpCandidates
    int trials = kTrials;
    bool failed = false;
    cudaEvent_t ev[kTrials][2] = {};
  };

  // Entry of `key`, created with its events on first use with `rounds` trial
  // rounds (1..kMaxRounds; rounds = 0 only looks up). nullptr when absent and
  // not created, the table is full, or events cannot be created: then
  // candidate 0 is used.
  Entry* find(uint64_t key, int rounds) {
    for (Entry& e : entries_)
      if (e.key == key) return &e;
    if (rounds < 1 || entries_.size() >= kMaxEntries) return nullptr;
    Entry e;
    e.key = key;
    e.trials = (rounds < kMaxRounds ? rounds : kMaxRounds) * kTwoOpCandidates;
    for (auto& pair : e.ev)
      for (cudaEvent_t& ev : pair)
        if (const cudaError_t ec = cudaEventCreate(&ev); ec != cudaSuccess) {
          clear_own_error(ec);
          e.chosen = 0;
        }
    entries_.push_back(e);
    return &entries_.back();
  }

  void decide(Entry& e) {
    if (e.failed) {
      e.chosen = 0;
      return;
    }
    if (e.next < e.trials) return;
    float best[kTwoOpCandidates];
    for (int i = 0; i < e.trials; ++i) {
      if (const cudaError_t q = cudaEventQuery(e.ev[i][1]); q != cudaSuccess) {  // not done yet (or failed)
        clear_own_error(q);
        return;
      }
      float ms = 0.0f;
      if (const cudaError_t t = cudaEventElapsedTime(&ms, e.ev[i][0], e.ev[i][1]); t != cudaSuccess) {
        clear_own_error(t);
        e.chosen = 0;
        return;
      }
      const int c = i % kTwoOpCandidates;
      if (i < kTwoOpCandidates || ms < best[c]) best[c] = ms;  // shortest of its rounds
    }
    int arg = 0;
    for (int c = 1; c < kTwoOpCandidates; ++c)
      if (best[c] < best[arg]) arg = c;
    e.chosen = arg;
  }

  static constexpr size_t kMaxEntries = 64;
  std::mutex mu_;
  std::vector<Entry> entries_;
};
TwoOpTuner g_two_op_tuner;

// Hash of what decides the two-op pass's speed: device, sizes, dtypes,
// 32-byte alignment (an FNV-style multiply-xor per 64-bit word, then a final
// avalanche; a collision only shares a tuning decision).
uint64_t list_key(const zo_tensor* params, int32_t n) {
  uint64_t h = 0xcbf29ce484222325ull;
  auto mix = [&h](uint64_t v) {
    h ^= v;
    h *= 0x100000001b3ull;
    h ^= h >> 29;
  };
  int dev = 0;
  cudaGetDevice(&dev);
  mix(static_cast<uint64_t>(dev));
  mix(static_cast<uint64_t>(n));
  for (int32_t t = 0; t < n; ++t) {
    mix(static_cast<uint64_t>(params[t].numel));
    mix(static_cast<uint64_t>(params[t].dtype) | (reinterpret_cast<uintptr_t>(params[t].ptr) % 32 == 0 ? 0x100u : 0u));
  }
  h ^= h >> 33;
  h *= 0xff51afd7ed558ccdull;
  h ^= h >> 33;
  return h;
}

// Enqueue perturb launches over the whole parameter list.
// Tensors of a perturb launch that are not 32-byte aligned go to
// perturb_shift_kernel: flag them (kShift). Returns a bit mask of their
// storage types; *main_work tells whether any other tensor has elements.
unsigned mark_shift(zo::TensorTable& tab, bool* main_work) {
  unsigned types = 0;
  *main_work = false;
  for (int i = 0; i < tab.n; ++i) {
    if (tab.numel[i] == 0) continue;
    if (tab.flags[i] & zo::kVec32) {
      *main_work = true;
    } else {
      tab.flags[i] |= zo::kShift;
      types |= 1u << (tab.flags[i] & zo::kDtypeMask);
    }
  }
  return types;
}

// grp_end over the flagged tensors of storage type dt (the others own no
// group). Returns the number of groups.
uint32_t shift_groups(const zo::TensorTable& tab, uint8_t dt, uint32_t* grp_end) {
  uint32_t groups = 0;
  for (int i = 0; i < tab.n; ++i) {
    const uint8_t fl = tab.flags[i];
    if ((fl & zo::kShift) && (fl & zo::kDtypeMask) == dt) {
      const uint32_t esz = dt == zo::kF32 ? 4 : 2;
      const int64_t a = static_cast<int64_t>(tab.ptr[i] % 32) / esz;  // 1..15: pointers are element-aligned
      const int64_t chunks = (tab.numel[i] + a + 15) / 16;
      groups += static_cast<uint32_t>((chunks + zo::kShiftGroup - 1) / zo::kShiftGroup);
    }
    grp_end[i] = groups;
  }
  return groups;
}

thread_local zo::ShiftParams tl_shift;
thread_local zo::UpdateShiftParams tl_update_shift;

int run_perturb(const zo_tensor* params, int32_t n, PerturbParams& pp, DeviceInfo* d, cudaStream_t s) {
  int loop = zo::kLoopBlocks, bps = d->perturb_bps, slot = -1;
  uint64_t key = 0;
  if (pp.nops == 2) {
    // probes in two groups of 8 (two Philox calls per block) run a kernel of
    // their own, so they get a configuration choice of their own, timed one
    // round per candidate: such calls come once per 8 probes, and three
    // rounds would leave a K = 16 step still timing candidates after a few
    // steps
    const bool cross = pp.op[0].ctr2 != pp.op[1].ctr2;
    key = list_key(params, n) ^ (cross ? 0x9E3779B97F4A7C15ull : 0ull);
    const int c = g_two_op_tuner.pick(key, cross ? 1 : 3, s, &slot);
    loop = kTwoOpLoop[c];
    bps = d->two_op_bps[c];
  }
  if (slot >= 0) g_two_op_tuner.record(key, slot, 0, s);
  int64_t blk = 0;
  for (int32_t t0 = 0; t0 < n;) {
    int64_t nb = 0;
    t0 = fill_table(pp.tab, params, t0, n, blk, &nb);
    if (nb > 0) {
      bool main_work = false;
      const unsigned shift_types = mark_shift(pp.tab, &main_work);
      bool f32v = false;  // aligned fp32 tensors in this launch: pipelined fp32 path (single-op kernel)
      for (int i = 0; i < pp.tab.n && !f32v; ++i)
        f32v = (pp.tab.flags[i] & zo::kVec32) && (pp.tab.flags[i] & zo::kDtypeMask) == zo::kF32;
      if (main_work) {
        cudaError_t e = zo::launch_perturb(pp, grid_for(pp.tab.blk_total, d->sms, bps), loop, f32v, s);
        if (e != cudaSuccess) return cuda_fail(e, "perturb_kernel");
      }
      if (shift_types) tl_shift.p = pp;
      for (uint8_t dt = 0; dt < 3; ++dt) {
        if (!(shift_types & (1u << dt))) continue;
        const uint32_t groups = shift_groups(pp.tab, dt, tl_shift.grp_end);
        tl_shift.grp_total = groups;
        const int64_t want = (static_cast<int64_t>(groups) * 32 + zo::kThreads - 1) / zo::kThreads;
        const int64_t cap = static_cast<int64_t>(d->sms) * d->shift_bps[pp.nops - 1][dt];
        cudaError_t e = zo::launch_perturb_shift(tl_shift, dt, static_cast<int>(want < cap ? want : cap), s);
        if (e != cudaSuccess) return cuda_fail(e, "perturb_shift_kernel");
      }
    }
    blk += nb;
  }
  if (slot >= 0) g_two_op_tuner.record(key, slot, 1, s);
  return ZO_OK;
}

// Fill a pair table with tensors t0, t0+1, ... (same split rules as
// fill_table).
int32_t fill_pair_table(zo::PairTable& tab, const zo_tensor* theta, const zo_tensor* plus, const zo_tensor* minus,
                        int32_t t0, int32_t n, int64_t blk_base, int64_t* nblocks) {
  tab.n = 0;
  tab.blk_base = blk_base;
  int64_t b = 0;
  int32_t t = t0;
  for (; t < n && tab.n < zo::kMaxTensorsPerLaunch; ++t) {
    const int64_t nb = (theta[t].numel + 15) / 16;
    if (tab.n > 0 && b + nb >= zo::kMaxLaunchBlocks) break;
    const int i = tab.n++;
    b += nb;
    tab.blk_end[i] = static_cast<uint32_t>(b);
    tab.src[i] = reinterpret_cast<uint64_t>(theta[t].ptr);
    tab.plus[i] = reinterpret_cast<uint64_t>(plus[t].ptr);
    tab.minus[i] = reinterpret_cast<uint64_t>(minus[t].ptr);
    tab.last[i] = static_cast<uint8_t>(theta[t].numel - 16 * (nb > 0 ? nb - 1 : 0));  // 1..16 (0 if empty)
    uint8_t fl = static_cast<uint8_t>(theta[t].dtype);
    if ((tab.src[i] | tab.plus[i] | tab.minus[i]) % 32 == 0) fl |= zo::kVec32;
    tab.flags[i] = fl;
  }
  tab.blk_total = static_cast<uint32_t>(b);
  *nblocks = b;
  return t;
}

// Tensors of a pair launch for pair_shift_kernel: fp32 tensors whose three
// pointers share their offset from the 32-byte grid, and 16-bit tensors not
// all 32-byte aligned whose plus and minus share theirs (theta may sit at
// another, the "moved" kernel); the others keep perturb_pair_kernel's paths.
// Returns a bit mask of (storage type, moved) classes: bit dt + 3 * moved.
bool pair_moved(const zo::PairTable& tab, int i) { return tab.src[i] % 32 != tab.plus[i] % 32; }

unsigned mark_pair_shift(zo::PairTable& tab, bool* main_work) {
  unsigned classes = 0;
  *main_work = false;
  for (int i = 0; i < tab.n; ++i) {
    const uint32_t begin = i == 0 ? 0u : tab.blk_end[i - 1];
    if (tab.blk_end[i] == begin) continue;  // empty
    const uint8_t dt = tab.flags[i] & zo::kDtypeMask;
    const bool outs = tab.plus[i] % 32 == tab.minus[i] % 32;
    const bool moved = pair_moved(tab, i);
    const bool take = dt == zo::kF32 ? (outs && !moved) : (outs && !(tab.flags[i] & zo::kVec32));
    if (take) {
      tab.flags[i] |= zo::kShift;
      classes |= 1u << (dt + 3 * (moved ? 1 : 0));
    } else {
      *main_work = true;
    }
  }
  return classes;
}

thread_local zo::PairShiftParams tl_pair_shift;

// Launch pair_shift_kernel over the flagged tensors of type dt whose theta
// is (moved) or is not at another offset than the outputs, in batches of
// kMaxPairShift entries.
int run_pair_shift(const zo::PairParams& pp, uint8_t dt, bool moved, DeviceInfo* d, cudaStream_t s) {
  zo::PairShiftParams& S = tl_pair_shift;
  S.keys = pp.keys;
  S.op = pp.op;
  const zo::PairTable& tab = pp.tab;
  const uint32_t esz = dt == zo::kF32 ? 4 : 2;
  int i = 0;
  while (i < tab.n) {
    S.n = 0;
    uint32_t groups = 0;
    for (; i < tab.n && S.n < zo::kMaxPairShift; ++i) {
      const uint8_t fl = tab.flags[i];
      if (!(fl & zo::kShift) || (fl & zo::kDtypeMask) != dt || pair_moved(tab, i) != moved) continue;
      const uint32_t begin = i == 0 ? 0u : tab.blk_end[i - 1];
      const int64_t numel = static_cast<int64_t>(tab.blk_end[i] - begin - 1) * 16 + tab.last[i];
      const int64_t a = static_cast<int64_t>(tab.plus[i] % 32) / esz;  // chunks follow the outputs
      const int64_t chunks = (numel + a + 15) / 16;
      const int j = S.n++;
      S.src[j] = tab.src[i];
      S.plus[j] = tab.plus[i];
      S.minus[j] = tab.minus[i];
      S.numel[j] = numel;
      S.vb0[j] = tab.blk_base + begin;
      groups += static_cast<uint32_t>((chunks + zo::kShiftGroup - 1) / zo::kShiftGroup);
      S.grp_end[j] = groups;
    }
    if (S.n == 0) break;
    S.grp_total = groups;
    const int64_t want = (static_cast<int64_t>(groups) * 32 + zo::kThreads - 1) / zo::kThreads;
    const int64_t cap = static_cast<int64_t>(d->sms) * kShiftBlocksPerSm;
    cudaError_t e = zo::launch_pair_shift(S, dt, moved, static_cast<int>(want < cap ? want : cap), s);
    if (e != cudaSuccess) return cuda_fail(e, "pair_shift_kernel");
  }
  return ZO_OK;
}

thread_local PerturbParams tl_perturb;
thread_local zo::PairParams tl_pair;
thread_local UpdateParams tl_update;

}  // namespace

extern "C" {

const char* zo_status_string(int status) {
  switch (status) {
    case ZO_OK: return "ZO_OK";
    case ZO_ERR_ARG: return "ZO_ERR_ARG: invalid argument";
    case ZO_ERR_DTYPE: return "ZO_ERR_DTYPE: unknown dtype";
    case ZO_ERR_ALIGN: return "ZO_ERR_ALIGN: pointer not aligned to its element size";
    case ZO_ERR_NONFINITE: return "ZO_ERR_NONFINITE: non-finite loss, curvature or coefficient";
    case ZO_ERR_CUDA: return "ZO_ERR_CUDA: CUDA runtime error";
    case ZO_ERR_TOO_MANY_PROBES: return "ZO_ERR_TOO_MANY_PROBES: K exceeds ZO_MAX_PROBES";
    case ZO_ERR_WORKSPACE: return "ZO_ERR_WORKSPACE: workspace missing or too small";
    default: return "unknown zo_status";
  }
}

const char* zo_last_cuda_error(void) { return g_last_cuda_error; }

int zo_version(void) { return 10400; }

int zo_set_packing(int32_t bits_per_value) {
  if (bits_per_value != zo::kPacking1 && bits_per_value != zo::kPacking8) return ZO_ERR_ARG;
  g_packing.store(bits_per_value);
  return ZO_OK;
}

int zo_get_packing(void) { return g_packing.load(); }

int zo_perturb(const zo_tensor* params, int32_t n_tensors, uint64_t seed, uint32_t probe, float scale,
               void* stream) {
  int packing = zo::kPacking1;
  int rc = validate_params(params, n_tensors, &packing);
  if (rc != ZO_OK) return rc;
  if (!std::isfinite(scale)) return ZO_ERR_ARG;
  if (n_tensors == 0) return ZO_OK;
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != ZO_OK) return rc;
  PerturbParams& pp = tl_perturb;
  pp.keys = expand_keys(seed);
  pp.probe = probe;
  pp.op[0] = make_op(probe, scale, packing);
  pp.op[1] = pp.op[0];
  pp.nops = 1;
  pp.coef = nullptr;
  pp.coef_mul = 0.0;
  pp.status = nullptr;
  return run_perturb(params, n_tensors, pp, d, static_cast<cudaStream_t>(stream));
}

int zo_perturb2(const zo_tensor* params, int32_t n_tensors, uint64_t seed, uint32_t probe_a, float scale_a,
                uint32_t probe_b, float scale_b, void* stream) {
  int packing = zo::kPacking1;
  int rc = validate_params(params, n_tensors, &packing);
  if (rc != ZO_OK) return rc;
  if (!std::isfinite(scale_a) || !std::isfinite(scale_b)) return ZO_ERR_ARG;
  if (n_tensors == 0) return ZO_OK;
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != ZO_OK) return rc;
  PerturbParams& pp = tl_perturb;
  pp.keys = expand_keys(seed);
  pp.probe = probe_a;
  pp.op[0] = make_op(probe_a, scale_a, packing);
  pp.op[1] = make_op(probe_b, scale_b, packing);
  pp.nops = 2;
  pp.coef = nullptr;
  pp.coef_mul = 0.0;
  pp.status = nullptr;
  return run_perturb(params, n_tensors, pp, d, static_cast<cudaStream_t>(stream));
}

int zo_perturb_pair(const zo_tensor* theta, const zo_tensor* plus, const zo_tensor* minus, int32_t n_tensors,
                    uint64_t seed, uint32_t probe, float scale, void* stream) {
  int packing = zo::kPacking1, pk_plus = 0, pk_minus = 0;
  int rc = validate_params(theta, n_tensors, &packing);
  if (rc != ZO_OK) return rc;
  if ((rc = validate_params(plus, n_tensors, &pk_plus)) != ZO_OK) return rc;
  if ((rc = validate_params(minus, n_tensors, &pk_minus)) != ZO_OK) return rc;
  // plus and minus follow theta's probes: they may name no packing or the same one
  if (n_tensors > 0 && ((plus[0].packing != 0 && pk_plus != packing) ||
                        (minus[0].packing != 0 && pk_minus != packing)))
    return ZO_ERR_ARG;
  if (!std::isfinite(scale)) return ZO_ERR_ARG;
  for (int32_t t = 0; t < n_tensors; ++t) {
    if (plus[t].numel != theta[t].numel || minus[t].numel != theta[t].numel) return ZO_ERR_ARG;
    if (plus[t].dtype != theta[t].dtype || minus[t].dtype != theta[t].dtype) return ZO_ERR_ARG;
    if (theta[t].numel > 0 && plus[t].ptr == minus[t].ptr) return ZO_ERR_ARG;
  }
  if (n_tensors == 0) return ZO_OK;
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != ZO_OK) return rc;
  zo::PairParams& pp = tl_pair;
  pp.keys = expand_keys(seed);
  pp.op = make_op(probe, scale, packing);
  int64_t blk = 0;
  for (int32_t t0 = 0; t0 < n_tensors;) {
    int64_t nb = 0;
    t0 = fill_pair_table(pp.tab, theta, plus, minus, t0, n_tensors, blk, &nb);
    if (nb > 0) {
      bool main_work = false;
      const unsigned shift_types = mark_pair_shift(pp.tab, &main_work);
      if (main_work) {
        cudaError_t e = zo::launch_perturb_pair(pp, grid_for(nb, d->sms, d->pair_bps),
                                                static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess) return cuda_fail(e, "perturb_pair_kernel");
      }
      for (unsigned cls = 0; cls < 6; ++cls) {
        if (!(shift_types & (1u << cls))) continue;
        const uint8_t dt = static_cast<uint8_t>(cls % 3);
        if ((rc = run_pair_shift(pp, dt, cls >= 3, d, static_cast<cudaStream_t>(stream))) != ZO_OK) return rc;
      }
    }
    blk += nb;
  }
  return ZO_OK;
}

static int check_update_args(const zo_tensor* params, int32_t n, const double* c, int32_t K, double lr,
                             int* packing) {
  int rc = validate_params(params, n, packing);
  if (rc != ZO_OK) return rc;
  if (K < 1) return ZO_ERR_ARG;
  if (K > ZO_MAX_PROBES) return ZO_ERR_TOO_MANY_PROBES;
  if (c == nullptr || !std::isfinite(lr)) return ZO_ERR_ARG;
  return ZO_OK;
}

int zo_update(const zo_tensor* params, int32_t n_tensors, uint64_t seed, const double* c, int32_t K, double lr,
              const int32_t* status, void* stream) {
  return zo_update_ex(params, n_tensors, seed, c, K, lr, status, 0, 0u, 0.0f, stream);
}

int zo_update_ex(const zo_tensor* params, int32_t n_tensors, uint64_t seed, const double* c, int32_t K, double lr,
                 const int32_t* status, int32_t has_pre, uint32_t pre_probe, float pre_scale, void* stream) {
  int packing = zo::kPacking1;
  int rc = check_update_args(params, n_tensors, c, K, lr, &packing);
  if (rc != ZO_OK) return rc;
  if (has_pre != 0 && !std::isfinite(pre_scale)) return ZO_ERR_ARG;
  if (n_tensors == 0) return rc;
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != ZO_OK) return rc;
  UpdateParams& up = tl_update;
  up.keys = expand_keys(seed);
  up.coef = c;
  up.coef_mul = -(lr / static_cast<double>(K));
  up.K = K;
  up.groups = (K + 7) / 8;
  up.packing = packing;
  up.has_pre = has_pre != 0;
  up.pre = make_op(pre_probe, has_pre != 0 ? pre_scale : 0.0f, up.packing);
  up.status = status;
  const bool lut8 = zo::lut8_supported(up.groups, up.packing) && up.groups >= kLut8MinGroups;
  int bps = 1;
  if (lut8) {
    if ((rc = lut8_blocks_per_sm(d, up.groups, &bps)) != ZO_OK) return rc;
  } else if ((rc = update_blocks_per_sm(d, up.groups, up.packing, &bps)) != ZO_OK) {
    return rc;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int64_t blk = 0;
  for (int32_t t0 = 0; t0 < n_tensors;) {
    int64_t nb = 0;
    t0 = fill_table(up.tab, params, t0, n_tensors, blk, &nb);
    if (nb > 0) {
      bool main_work = false;
      const unsigned shift_types = mark_shift(up.tab, &main_work);
      if (main_work && lut8) {
        cudaError_t e = zo::launch_update_lut8(up, d->sms, bps, s);
        if (e != cudaSuccess) return cuda_fail(e, "update_lut8_kernel");
      } else if (main_work) {
        cudaError_t e = zo::launch_update(up, grid_for(up.tab.blk_total, d->sms, bps * kUpdateWaves), s);
        if (e != cudaSuccess) return cuda_fail(e, "update_kernel");
      }
      if (shift_types) tl_update_shift.u = up;
      for (uint8_t dt = 0; dt < 3; ++dt) {
        if (!(shift_types & (1u << dt))) continue;
        const uint32_t groups = shift_groups(up.tab, dt, tl_update_shift.grp_end);
        tl_update_shift.grp_total = groups;
        int sbps = 1;
        if ((rc = update_shift_blocks_per_sm(d, up.groups, up.packing, dt, &sbps)) != ZO_OK) return rc;
        const int64_t want = (static_cast<int64_t>(groups) * 32 + zo::kThreads - 1) / zo::kThreads;
        const int64_t cap = static_cast<int64_t>(d->sms) * sbps * kUpdateWaves;
        cudaError_t e = zo::launch_update_shift(tl_update_shift, dt, static_cast<int>(want < cap ? want : cap), s);
        if (e != cudaSuccess) return cuda_fail(e, "update_shift_kernel");
      }
    }
    blk += nb;
  }
  return ZO_OK;
}

int zo_update_sequential(const zo_tensor* params, int32_t n_tensors, uint64_t seed, const double* c, int32_t K,
                         double lr, const int32_t* status, void* stream) {
  int packing = zo::kPacking1;
  int rc = check_update_args(params, n_tensors, c, K, lr, &packing);
  if (rc != ZO_OK || n_tensors == 0) return rc;
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != ZO_OK) return rc;
  PerturbParams& pp = tl_perturb;
  pp.keys = expand_keys(seed);
  pp.coef = c;
  pp.coef_mul = -(lr / static_cast<double>(K));
  pp.status = status;
  pp.nops = 1;
  for (int32_t k = 0; k < K; ++k) {
    pp.probe = static_cast<uint32_t>(k);
    pp.op[0] = make_op(pp.probe, 0.0f, packing);  // scale read from c on the device
    pp.op[1] = pp.op[0];
    if ((rc = run_perturb(params, n_tensors, pp, d, static_cast<cudaStream_t>(stream))) != ZO_OK) return rc;
  }
  return ZO_OK;
}

static int check_precondition_args(const double* losses, int32_t K, double eps, double alpha, double lambda_reg,
                                   const double* c, const int32_t* status) {
  if (K < 1) return ZO_ERR_ARG;
  if (K > ZO_MAX_PROBES) return ZO_ERR_TOO_MANY_PROBES;
  if (losses == nullptr || c == nullptr || status == nullptr) return ZO_ERR_ARG;
  if (!(eps > 0.0) || !std::isfinite(eps)) return ZO_ERR_ARG;
  if (!(alpha >= 0.0) || !(alpha <= 1.0)) return ZO_ERR_ARG;
  if (!(lambda_reg > 0.0) || !std::isfinite(lambda_reg)) return ZO_ERR_ARG;
  return ZO_OK;
}

int zo_precondition_ex(const double* losses, int32_t K, double eps, double alpha, double lambda_reg,
                       int32_t flags, double* c, double* w, double* curv, int32_t* status, void* stream) {
  int rc = check_precondition_args(losses, K, eps, alpha, lambda_reg, c, status);
  if (rc != ZO_OK) return rc;
  if ((flags & ~(ZO_PRECOND_ONE_SIDED | ZO_PRECOND_RELATIVE_CURVATURE)) != 0) return ZO_ERR_ARG;
  static_assert(ZO_PRECOND_ONE_SIDED == zo::kPrecondOneSided && ZO_PRECOND_RELATIVE_CURVATURE == zo::kPrecondRelative,
                "flag values");
  cudaError_t e = zo::launch_precondition(losses, K, eps, alpha, lambda_reg, flags, c, w, curv, status,
                                          static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ZO_OK : cuda_fail(e, "precondition_kernel");
}

int zo_precondition(const double* losses, int32_t K, double eps, double* c, int32_t* status, void* stream) {
  return zo_precondition_ex(losses, K, eps, 0.1, 1.0, 0, c, nullptr, nullptr, status, stream);
}

static int probe_view_grid(int64_t blocks, int* grid) {
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != ZO_OK) return rc;
  *grid = grid_for(blocks, d->sms, 8);
  return ZO_OK;
}

int zo_probe_bytes(uint64_t seed, uint32_t probe, int64_t first, int64_t n, uint8_t* out, void* stream) {
  if (first < 0 || n < 0 || (n > 0 && out == nullptr)) return ZO_ERR_ARG;
  if (n > (INT64_C(1) << 58) - first) return ZO_ERR_ARG;
  if (n == 0) return ZO_OK;
  int grid = 1;
  int rc = probe_view_grid((n + 1) / 2 + 1, &grid);
  if (rc != ZO_OK) return rc;
  uint32_t ctr2 = 0, bit = 0;
  probe_counter(probe, g_packing.load(), &ctr2, &bit);
  cudaError_t e = zo::launch_probe_bytes(expand_keys(seed), ctr2, bit, first, n, out, grid,
                                         static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ZO_OK : cuda_fail(e, "probe_bytes_kernel");
}

int zo_probe_signs(uint64_t seed, uint32_t probe, int64_t first, int64_t n, int8_t* out, void* stream) {
  if (first < 0 || n < 0 || (n > 0 && out == nullptr)) return ZO_ERR_ARG;
  if (n > (INT64_C(1) << 58) - first) return ZO_ERR_ARG;
  if (n == 0) return ZO_OK;
  int grid = 1;
  int rc = probe_view_grid(n / 16 + 2, &grid);
  if (rc != ZO_OK) return rc;
  uint32_t ctr2 = 0, bit = 0;
  probe_counter(probe, g_packing.load(), &ctr2, &bit);
  cudaError_t e = zo::launch_probe_signs(expand_keys(seed), ctr2, bit, first, n, out, grid,
                                         static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ZO_OK : cuda_fail(e, "probe_signs_kernel");
}

int64_t zo_quadratic_loss_workspace_size(int64_t n) {
  (void)n;
  return static_cast<int64_t>(zo::kMaxLossPartials) * static_cast<int64_t>(sizeof(double));
}

int zo_quadratic_loss(const float* theta, const float* a, int64_t n, double* out, void* workspace,
                      int64_t workspace_bytes, void* stream) {
  if (n < 0 || out == nullptr || (n > 0 && (theta == nullptr || a == nullptr))) return ZO_ERR_ARG;
  if (workspace == nullptr || workspace_bytes < zo_quadratic_loss_workspace_size(n)) return ZO_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % sizeof(double) != 0) return ZO_ERR_ALIGN;
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != ZO_OK) return rc;
  cudaError_t e = zo::launch_quadratic_loss(theta, a, n, out, static_cast<double*>(workspace), zo::kMaxLossPartials,
                                            d->sms, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ZO_OK : cuda_fail(e, "quadratic_loss");
}

int64_t zo_perturb_quadratic_loss_workspace_size(int64_t n) {
  (void)n;
  // the partials, then the ticket counter (8 bytes keep the size a multiple of 8)
  return static_cast<int64_t>(zo::kMaxQuadPassPartials) * static_cast<int64_t>(sizeof(double)) + 8;
}

int zo_perturb_quadratic_loss(float* theta, const float* a, int64_t n, uint64_t seed, int32_t packing, int32_t nops,
                              uint32_t probe_a, float scale_a, uint32_t probe_b, float scale_b, double* out,
                              int32_t out_copies, int64_t out_stride, void* workspace, int64_t workspace_bytes,
                              void* stream) {
  if (n < 0 || out == nullptr || (n > 0 && (theta == nullptr || a == nullptr))) return ZO_ERR_ARG;
  if (nops < 0 || nops > 2 || out_copies < 1 || out_stride < 1) return ZO_ERR_ARG;
  if (packing != 0 && packing != zo::kPacking1 && packing != zo::kPacking8) return ZO_ERR_ARG;
  if ((nops >= 1 && !std::isfinite(scale_a)) || (nops == 2 && !std::isfinite(scale_b))) return ZO_ERR_ARG;
  if (reinterpret_cast<uintptr_t>(theta) % sizeof(float) != 0 || reinterpret_cast<uintptr_t>(a) % sizeof(float) != 0)
    return ZO_ERR_ALIGN;
  if (workspace == nullptr || workspace_bytes < zo_perturb_quadratic_loss_workspace_size(n)) return ZO_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(workspace) % sizeof(double) != 0) return ZO_ERR_ALIGN;
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != ZO_OK) return rc;
  const int pk = packing != 0 ? packing : g_packing.load();
  const zo::RoundKeys keys = expand_keys(seed);
  const zo::PerturbOp ops[2] = {make_op(probe_a, scale_a, pk), make_op(probe_b, scale_b, pk)};
  double* partial = static_cast<double*>(workspace);
  uint32_t* ticket = reinterpret_cast<uint32_t*>(partial + zo::kMaxQuadPassPartials);
  cudaError_t e = zo::launch_perturb_quad_loss(theta, a, n, keys, ops, nops, out, out_copies, out_stride, partial,
                                               ticket, zo::kMaxQuadPassPartials, d->sms,
                                               static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ZO_OK : cuda_fail(e, "perturb_quad_loss");
}

int zo_quadratic_loss_static(const float* theta, const float* a, int64_t n, double* out, void* stream) {
  if (n < 0 || out == nullptr || (n > 0 && (theta == nullptr || a == nullptr))) return ZO_ERR_ARG;
  if (n > ZO_QUADRATIC_LOSS_STATIC_MAX_N) return ZO_ERR_WORKSPACE;
  static_assert(ZO_QUADRATIC_LOSS_STATIC_MAX_N == zo::kStaticLossPartials * zo::kStaticLossSlice,
                "static scratch capacity and the documented limit must agree");
  cudaError_t e = zo::launch_quadratic_loss_static(theta, a, n, out, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? ZO_OK : cuda_fail(e, "quadratic_loss_static");
}

}  // extern "C"
