// Internal declarations shared by the AVTP CUDA translation units.
// Nothing here is part of the C ABI; see include/avtp.h for that.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <mutex>
#include <utility>

#include "avtp.h"

namespace avtp {

// ---------------------------------------------------------------- limits
constexpr int kMaxImagesPerRequest = 4096;
constexpr int kMaxVisualPerRequest = 1 << 20;
constexpr int kFxFracBits = 32;          // per-token fixed point of the per-image sums
constexpr float kFxScoreLimit = 1024.f;  // |score| clamp before the fixed-point conversion
constexpr int kRatioFracBits = 40;       // ratio grid of the budget rule
constexpr double kRatioLimit = 1048576.0;  // ratios saturate at +-2^20 before the grid

// Tiles of the text-attention criterion (tensor-core path). Rows are (text query, head
// of the KV group) pairs, G = Hq / Hkv of them per text query, in text order. A request's
// rows are cut into blocks of kAttnBlockRows; pass 1 runs a block as two MMA A tiles
// against key tiles of kAttnTileN keys, pass 2 holds a block as the MMA B operand and
// streams key tiles of kAttnTileM visual keys through it.
constexpr int kAttnTileM = 128;          // MMA M: rows of a pass-1 A tile, keys of a pass-2 tile
constexpr int kAttnTileN = 256;          // MMA N: keys per pass-1 step, rows of a pass-2 block
constexpr int kAttnBlockRows = 256;      // rows per block (both passes)
constexpr int kAttnMaxChunks = 64;       // pass-1 partial (max, sum) slots per row at most
constexpr int kAttnMaxGroupHeads = 128;  // Hq / Hkv at most
constexpr int kAttnMassFracBits = 40;    // fixed point of the per-key probability mass

// ---------------------------------------------------------------- status
// First word of every workspace. code: first error recorded (0 = none);
// layout_ok: set by the validation kernel when the layout may be used.
struct DevStatus {
  int32_t code;
  int32_t layout_ok;
  int32_t detail;  // index of the first offending item, for debugging
  uint32_t pool;   // tokens the criterion-A scoring kernel's warps have drawn from its pool
};

__device__ __forceinline__ void record_error(DevStatus* st, int32_t code, int32_t detail) {
  if (atomicCAS(&st->code, 0, code) == 0) st->detail = detail;
}

// ---------------------------------------------------------------- bounded waits
// Every wait on an mbarrier gives up after about kWaitLimitNs of the global timer
// without the phase completing (or after kWaitSpinCap polls, should the timer not
// advance); the kernel then records AVTP_ERR_TIMEOUT and returns instead of hanging.
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // one second
constexpr uint32_t kWaitSpinCap = 1u << 28;

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Called after each failed poll (polls counts them from 1): true once the wait has run
// past limit_ns. The timer is read every 64 polls only, and started at the first such
// read, so that the short waits of a running pipeline never touch it.
__device__ __forceinline__ bool wait_expired(uint32_t polls, uint64_t& t0, uint64_t limit_ns) {
  if ((polls & 63u) != 0) return false;
  const uint64_t now = global_ns();
  if (polls == 64) {
    t0 = now;
    return false;
  }
  return now - t0 > limit_ns || polls >= kWaitSpinCap;
}

// ---------------------------------------------------------------- phase timeline (diagnostic build)
// Built with -DAVTP_TIMELINE, the kernels of the fused stage record global-timer stamps of
// their phases in the bytes between the workspace's status word and its first array
// (every workspace slice is 256-byte aligned, so 240 bytes are free there): for every
// event the earliest stamp over the CTAs that reach it (first kTlEvents words) and the
// latest (next kTlEvents words). avtp_prune presets those words before its first kernel.
// The normal build records nothing and never touches them.
enum TimelineEvent {
  kTlPrepBegin = 0, kTlPrepEnd, kTlScoreBegin, kTlScoreEnd, kTlSelBegin, kTlSelDryEnd, kTlSelWaited, kTlRuleBegin,
  kTlRuleEnd, kTlSelEnd, kTlCompactBegin, kTlCompactWaited, kTlCompactEnd, kTlHistDone, kTlEvents
};
constexpr size_t kTimelineOffset = 16;  // bytes after the start of the workspace
static_assert(kTimelineOffset + 2 * kTlEvents * sizeof(uint64_t) <= 256, "timeline must fit before the first array");

__device__ __forceinline__ void timeline_stamp(DevStatus* st, int ev) {
#ifdef AVTP_TIMELINE
  unsigned long long* tl = reinterpret_cast<unsigned long long*>(reinterpret_cast<char*>(st) + kTimelineOffset);
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  atomicMin(tl + ev, t);
  atomicMax(tl + kTlEvents + ev, t);
#else
  (void)st;
  (void)ev;
#endif
}

// The last of a CTA's nwarps warps to call it stamps ev, so that a CTA sends one pair of
// atomics to the timeline words, not one per warp (thousands of same-address atomics at
// the end of a kernel would queue behind each other and move the stamps). *count starts
// at zero (the caller clears it and synchronises the CTA before the first call).
__device__ __forceinline__ void timeline_stamp_cta(DevStatus* st, int ev, unsigned* count, unsigned nwarps) {
#ifdef AVTP_TIMELINE
  __syncwarp();
  if ((threadIdx.x & 31) == 0 && atomicAdd(count, 1u) == nwarps - 1) timeline_stamp(st, ev);
#else
  (void)st;
  (void)ev;
  (void)count;
  (void)nwarps;
#endif
}

// ---------------------------------------------------------------- workspace
struct WsPlan {
  size_t status;      // DevStatus
  size_t vis_cu;      // int32 [n_img + 1]: exclusive prefix of img_len over all images
  size_t img_req;     // int32 [n_img]: request of each image
  size_t req_budget;  // int32 [R]: B_r
  size_t img_sums;    // int64 [n_img]: used by avtp_prune when the caller passes NULL
  size_t scores;      // float [T]: used by avtp_prune when the caller passes NULL
  size_t scratch;     // int32 [n_img + 1]: per-call scratch of the pruned-layout kernel
  // criterion B (text attention); "rows" = rows per KV group = max_text * G
  size_t text_idx;    // int32 [T]: packed position of each text ordinal
  size_t text_cu;     // int32 [R + 1]: text ordinals per request
  size_t blk_cu;      // int32 [R + 1]: row blocks per request
  size_t p1s_cu;      // int32 [n_blocks_max + 1]: pass-1 key steps per row block
  size_t p2t_cu;      // int32 [n_blocks_max + 1]: pass-2 key tiles per row block
  size_t ktile_cu;    // int32 [n_img + 1]: key tiles per image
  size_t ktile_img;   // int32 [n_ktiles_max]: image of every key tile
  size_t meta;        // int32 [8]: F1, C1, F2, C2 (flat pass lengths per KV group, steps per CTA)
  size_t qt;          // bf16 [Hkv, rows, d]: the text queries, packed by KV group
  size_t lse_rows;    // float [Hkv, rows]: log2-domain LSE of every row (supplied LSE only)
  size_t p1_part;     // float2 [Hkv * n_blocks_max][256][kAttnMaxChunks]: per-CTA (max, sum) of every row
  size_t mass;        // uint64 [n_ktiles_max][128]: fixed-point probability mass of every visual key, by key tile
  size_t zbuf;        // float: the CUDA-core path's logits, request by request [its rows][its tokens]
  size_t total;
};

// Sizes of the text-attention bookkeeping that the host fixes before launch.
struct AttnPlan {
  int G;                 // query heads per KV group
  int64_t max_text;      // text tokens of the whole batch, at most
  int64_t rows;          // rows per KV group: max_text * G
  int64_t n_blocks_max;  // row blocks of all requests, at most
  int64_t n_ktiles_max;  // key tiles of all images, at most
  int Hkv;               // KV groups
  int grid;              // CTAs of the persistent tensor-core kernels (one per SM)
};
AttnPlan attn_plan(const avtp_layout_t& L, const avtp_score_args_t& sa);

// The CUDA-core path of criterion B (k_score_narrow.cu): rows are the batch's queries (at
// most) times Hq; the logits pass splits every (request, KV group) into NS key ranges and
// keeps every logit, Hq x queries x tokens of each request, at most kNarrowMaxLogitBytes.
constexpr int kNarrowMaxSplits = 64;
constexpr int64_t kNarrowMaxLogitBytes = int64_t(1) << 30;
// AVTP_PATH_AUTO takes the CUDA cores for AVTP_QUERIES_LAST, and for AVTP_QUERIES_TEXT
// only when the batch has at most this many rows per KV group (decided from its text-token
// bound). Measured on a request of four 640-token images and Qwen3-shaped heads (8 KV
// groups of 4 heads, d = 128), score call event-timed: 29.3 us on the narrow path against
// 34.4 us on tcgen05 at 4 rows per group (one text token), 33.4 against 34.4 at 8, and
// the narrow path growing with the rows beyond (tcgen05 stays near 33 us up to 256 rows).
constexpr int64_t kNarrowAutoRows = 4;
struct NarrowPlan {
  int G;
  int64_t rows;     // global rows (query ordinal x Hq + head), at most
  int NS;
  int64_t z_elems;  // logits, at most
};
NarrowPlan narrow_plan(const avtp_layout_t& L, const avtp_score_args_t& sa, int64_t max_text);
bool attn_uses_cuda_cores(const avtp_layout_t& L, const avtp_score_args_t& sa);

WsPlan plan_workspace(const avtp_layout_t& L, const avtp_score_args_t* sa);

template <typename T>
__host__ __device__ __forceinline__ T* ws_at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

// ---------------------------------------------------------------- parameter domain
// True when v * 2^32 is an integer: the budget rule takes alpha, the clamps and the keep
// ratios as exact multiples of 2^-32 (every fp32 value of at least 2^-9 is one).
__host__ __device__ __forceinline__ bool multiple_of_2m32(float v) {
  uint32_t b;
  memcpy(&b, &v, sizeof b);
  const int e8 = static_cast<int>((b >> 23) & 0xffu);
  const uint32_t mant = b & 0x7fffffu;
  if (e8 == 0) return mant == 0;  // zero; a subnormal is below 2^-126
  const int sh = e8 - 150 + 32;   // v * 2^32 = (mant + 2^23) * 2^sh
  if (sh >= 0) return true;
  if (sh <= -24) return false;
  return ((mant | 0x800000u) & ((1u << -sh) - 1u)) == 0;
}

// ---------------------------------------------------------------- small device helpers
__device__ __forceinline__ int64_t fixed_point_score(float s) {
  // rint(fx(s) * 2^32) with fx: NaN -> 0, clamp to [-2^10, 2^10], rounding half to
  // even. Done on the fp32 bits with integer operations (fp64 is scarce on this
  // part): s = M * 2^e with a 24-bit integer M, so s * 2^32 = M * 2^(e + 32).
  if (isnan(s)) return 0;
  s = fminf(fmaxf(s, -kFxScoreLimit), kFxScoreLimit);
  const uint32_t b = __float_as_uint(s);
  const int biased = static_cast<int>((b >> 23) & 0xFFu);
  if (biased == 0) return 0;  // zero or subnormal: |s * 2^32| < 2^-94
  const int64_t M = static_cast<int64_t>((b & 0x7FFFFFu) | 0x800000u);
  const int sh = biased - 127 - 23 + 32;  // s * 2^32 = M * 2^sh, sh <= 19 after the clamp
  int64_t v;
  if (sh >= 0) {
    v = M << sh;
  } else if (-sh > 25) {
    v = 0;  // M * 2^sh < 1/2
  } else {
    const int rs = -sh;
    const int64_t q = M >> rs, rem = M & ((int64_t(1) << rs) - 1), half = int64_t(1) << (rs - 1);
    v = q + ((rem > half || (rem == half && (q & 1))) ? 1 : 0);
  }
  return (b >> 31) ? -v : v;
}

// Order-preserving key: larger score -> larger key; NaN -> 0 (below -inf); -0 == +0.
__device__ __forceinline__ uint32_t rank_key(float s) {
  if (isnan(s)) return 0u;
  uint32_t b = __float_as_uint(s);
  if (b == 0x80000000u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Largest r in [0, n) with a[r] <= v, for non-decreasing a[0..n] with a[0] <= v.
__device__ __forceinline__ int upper_index(const int32_t* a, int n, int64_t v) {
  int lo = 0, hi = n;  // a[lo] <= v; answer in [lo, hi)
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (static_cast<int64_t>(a[mid]) <= v) lo = mid; else hi = mid;
  }
  return lo;
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// ---------------------------------------------------------------- programmatic dependent launch
// A kernel launched with programmatic stream serialization may start before the
// kernel ahead of it in the stream has finished. It must call pdl_wait() before
// it reads anything that kernel writes, and every thread calls it before exiting,
// so that the completion of a grid implies the completion of all grids before it.
// pdl_trigger() lets the next grid in the stream be scheduled. Without the launch
// attribute both are no-ops.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// True unless the environment sets AVTP_PDL=0 (read once).
bool pdl_enabled();

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl,
                          Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  const bool use = pdl && pdl_enabled();
  cfg.attrs = use ? attr : nullptr;
  cfg.numAttrs = use ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------- per-device set-up
// CUDA keeps function attributes (shared-memory size, carveout) per device, so a process
// that runs the library on several devices must set them on each. PerDevice records, per
// device ordinal, that a set-up succeeded (and an int it computed), under a lock.
constexpr int kMaxDevices = 64;
struct PerDevice {
  std::mutex mu;
  bool done[kMaxDevices] = {};
  int value[kMaxDevices] = {};
};

// Runs fn(dev, &value) for the current device unless it already succeeded there; returns
// its error. *out (optional) receives the value it stored.
template <class F>
cudaError_t once_per_device(PerDevice& pd, F&& fn, int* out = nullptr) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) {
    int v = 0;
    e = fn(dev, &v);
    if (out != nullptr) *out = v;
    return e;
  }
  std::lock_guard<std::mutex> lock(pd.mu);
  if (!pd.done[dev]) {
    e = fn(dev, &pd.value[dev]);
    if (e != cudaSuccess) return e;
    pd.done[dev] = true;
  }
  if (out != nullptr) *out = pd.value[dev];
  return cudaSuccess;
}

// ---------------------------------------------------------------- launchers (one per kernel)
struct PrepArgs {
  avtp_layout_t L;
  const float* keep_ratio;   // NULL: no budgets / out_cu_seqlens
  float r_min, r_max;        // each keep ratio must lie in [r_min, r_max]
  int32_t* out_cu_seqlens;   // NULL: not written
  int64_t* zero_img_sums;    // NULL: not zeroed
  int build_text_tiles;      // criterion B bookkeeping, sized by `attn`
  AttnPlan attn;
  // The image spans of the pruned batch (avtp_pruned_layout), from these budgets; NULL: none.
  const int32_t* pl_budgets;
  int32_t* pl_out_start;
  int32_t* pl_out_len;
};
cudaError_t launch_prep(const PrepArgs& a, void* ws, const WsPlan& p, cudaStream_t s);

// reserve_sms: SMs left free for the next kernel of the fused stage (see prune_reserve_sms).
cudaError_t launch_score_hvar(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                              int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s, int reserve_sms = 0);

cudaError_t launch_score_attn(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                              int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s);
cudaError_t launch_score_narrow(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores, int64_t* img_sums,
                                void* ws, const WsPlan& p, const AttnPlan& plan, cudaStream_t s);
// Scores and fixed-point image sums from the per-key mass of either criterion-B path.
cudaError_t launch_attn_finalize(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                                 int64_t* img_sums, void* ws, const WsPlan& p, const AttnPlan& plan, cudaStream_t s);

cudaError_t launch_allocate(const avtp_layout_t& L, const int64_t* img_sums, const avtp_alloc_args_t& aa,
                            int32_t* budgets, void* ws, const WsPlan& p, cudaStream_t s);

cudaError_t launch_select(const avtp_layout_t& L, const float* scores, const int32_t* budgets,
                          const int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, void* ws,
                          const WsPlan& p, cudaStream_t s);

// Budget rule and selection in one kernel (the fused stage). Its first warm_ctas CTAs
// run the code once on made-up data before waiting for the scores (see prune_reserve_sms).
cudaError_t launch_alloc_select(const avtp_layout_t& L, const int64_t* img_sums, const avtp_alloc_args_t& aa,
                                int32_t* budgets, const float* scores, const int32_t* out_cu_seqlens,
                                int32_t* kept_idx, int64_t n_kept, void* ws, const WsPlan& p, cudaStream_t s,
                                int warm_ctas = 0);

// In avtp_prune with the hidden-variation criterion on a small batch, the scoring
// kernel leaves prune_reserve_sms(L) SMs free so that the selection kernel's CTAs (one
// per image and one per request, one per SM) start while the scores stream in and warm
// their instruction caches (prune_warm_ctas(L) of them run the code once on made-up data
// first); 0 otherwise. Right after the scoring stream has swept L2 a cold run of the
// budget rule and the selection takes several times longer. On large batches the
// scoring time would grow instead.
constexpr int kMaxWarmCtas = 96;
int prune_reserve_sms(const avtp_layout_t& L);
int prune_warm_ctas(const avtp_layout_t& L);


cudaError_t launch_compact(const int32_t* kept_idx, int64_t n_kept, int64_t n_tokens, const avtp_rows_t* sets,
                           int n_sets, void* ws, const WsPlan& p, cudaStream_t s);

cudaError_t launch_wait_selftest(uint64_t limit_ns, int arrive, void* ws, cudaStream_t s);

cudaError_t launch_layer_attention(const avtp_layout_t& L, const int64_t* img_sums, int64_t* A, int n_layers,
                                   int layer, void* ws, const WsPlan& p, cudaStream_t s);
cudaError_t launch_layer_select(const int64_t* A, int n_samples, int n_layers, int k, int64_t* rank_sum,
                                int32_t* top_layers, cudaStream_t s);

int device_sm_count();

}  // namespace avtp
