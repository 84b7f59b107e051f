// Step 3: per-image top-k, text always kept, positions emitted in ascending order
// (paper §3.1: the pruned sequence is an order-preserving subsequence; §3.3.3:
// image i keeps its k_i most important tokens).
//
// One CTA (8 warps) per image, plus one per request for the text before its
// first image. Ranking uses order-preserving 32-bit keys (score descending, NaN
// lowest, -0 == +0) with ties to the lower position. A radix select finds the
// k-th key K*: the passes start below the highest bit in which the image's keys
// differ, use 8-bit digits with per-warp sub-histograms (no contention between
// warps), and stop as soon as the chosen digit's candidates are all kept. Tokens
// above K* are kept, and of those equal to K* the first k - #{key > K*} by
// position; kept positions are written in order after two block scans. The CTA
// also writes the text run that follows its image.
//
// Two kernels: k_select takes the budgets as input (avtp_select); k_alloc_select
// runs the budget rule of avtp_alloc.cuh for the image's request in warp 0 while
// warps 1-7 stage the keys and build the first histogram, then selects
// (avtp_prune). Everything that needs only the call's inputs is done before the
// kernel waits for the scoring kernel, so it overlaps the scoring.
#include "avtp_alloc.cuh"

namespace avtp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kPer = 8;                   // keys per thread in a tile
constexpr int kKeyCap = kThreads * kPer;  // keys staged in shared memory (2048)
constexpr unsigned kFull = 0xffffffffu;

struct SelectArgs {
  const int32_t* cu;
  const int32_t* icu;
  const int32_t* ist;
  const int32_t* iln;
  int R;
  int NI;
  int64_t T;
  const float* scores;
  const int32_t* out_cu;
  int32_t* kept_idx;
  int64_t n_kept;
  const int32_t* vis_cu;
  const int32_t* img_req;
  DevStatus* st;
};

struct SelShared {
  __align__(16) uint32_t keys[kKeyCap];
  int hist[kWarps][256];
  int wsum[kWarps];
  uint32_t wmin[kWarps], wmax[kWarps];
  int digit, above, count;
  // hand-over from the warps of the fused kernel
  uint32_t kmin, kmax;
  int k, before, total, alloc_err, out_lo, out_hi, vis_before, n_vis;
  int ncand;      // candidates gathered from the chosen first-pass bucket
  uint32_t thr;   // the k-th largest key, found among them
  // inputs of the fused kernel's warm-up run (see alloc_select_tail)
  int32_t dry_status[4];  // a status word that reads "layout ok"
  int32_t dry_out[2];
};

// Named barrier for warps 1..7 (224 threads) while warp 0 runs the budget rule.
__device__ __forceinline__ void bar_workers() { asm volatile("bar.sync 1, 224;" ::: "memory"); }

// Inclusive scan of v over the block in thread order; the block total goes to *total.
// Out of line: called several times per kernel, so its code is fetched once.
__device__ __noinline__ int block_incl_scan(int v, int* wsum, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();  // wsum may still be read by a previous scan
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  int pre = 0, tot = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    const int t = wsum[w];
    pre += w < warp ? t : 0;
    tot += t;
  }
  *total = tot;
  return pre + x;
}

struct KeySource {
  const float* sc;
  const uint32_t* staged;  // nullptr: read from global
  __device__ __forceinline__ uint32_t operator()(int j) const { return staged ? staged[j] : rank_key(sc[j]); }
};

// One histogram pass over the candidates (key & mask) == prefix, digit = (key >> shift) & dmask,
// into the calling warp's sub-histogram (cleared by the caller). Threads take keys tid, tid+nthreads, ...
__device__ __noinline__ void hist_pass(const KeySource& key_at, int n, uint32_t mask, uint32_t prefix, int shift,
                                          uint32_t dmask, int* my_hist, int tid, int nthreads) {
  for (int j = tid; j < n; j += nthreads) {
    const uint32_t key = key_at(j);
    if ((key & mask) == prefix) atomicAdd(&my_hist[(key >> shift) & dmask], 1);
  }
}

// From the sub-histograms, the digit holding the `remaining`-th largest candidate.
// All threads call; the answer is left in sh.digit / sh.above / sh.count.
__device__ __noinline__ void choose_digit(SelShared& sh, int remaining) {
  const int d = 255 - static_cast<int>(threadIdx.x);  // thread order = descending digits
  int c = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) c += sh.hist[w][d];
  int tot;
  const int incl = block_incl_scan(c, sh.wsum, &tot);
  const int excl = incl - c;
  if (excl < remaining && remaining <= incl) {
    sh.digit = d;
    sh.above = excl;
    sh.count = c;
  }
  __syncthreads();
}

__device__ __forceinline__ int highest_differing_bit(uint32_t kmin, uint32_t kmax) {
  return kmin == kmax ? -1 : 31 - __clz(kmin ^ kmax);
}
__device__ __forceinline__ uint32_t shared_bits_mask(int top) {
  return top < 0 ? 0xffffffffu : (top == 31 ? 0u : ~((2u << top) - 1u));
}

// Keep the top k of the n tokens whose scores start at sc (packed position t0), in
// ascending position order, at kept_idx[base ...]. kmin/kmax: range of the keys.
// With first_pass_done the sub-histograms already hold the first pass.
__device__ void block_select(const float* __restrict__ sc, int n, int k, int64_t t0, int64_t base,
                             int32_t* __restrict__ kept_idx, SelShared& sh, bool keys_staged, uint32_t kmin,
                             uint32_t kmax, bool first_pass_done) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (k >= n) {
    for (int j = tid; j < n; j += kThreads) kept_idx[base + j] = static_cast<int32_t>(t0 + j);
    return;
  }
  if (k <= 0) return;
  const KeySource key_at{sc, keys_staged ? sh.keys : nullptr};
  const int top = highest_differing_bit(kmin, kmax);
  uint32_t mask = shared_bits_mask(top);
  uint32_t prefix = kmin & mask;
  int remaining = k;
  bool have_hist = first_pass_done;
  for (int hi = top; hi >= 0; hi -= 8) {
    const int shift = hi >= 7 ? hi - 7 : 0;
    const uint32_t dmask = (2u << (hi - shift)) - 1u;
    if (!have_hist) {
#pragma unroll
      for (int q = 0; q < 8; ++q) sh.hist[warp][lane * 8 + q] = 0;
      __syncwarp();
      hist_pass(key_at, n, mask, prefix, shift, dmask, sh.hist[warp], tid, kThreads);
    }
    have_hist = false;
    __syncthreads();
    choose_digit(sh, remaining);
    prefix |= static_cast<uint32_t>(sh.digit) << shift;
    mask |= dmask << shift;
    remaining -= sh.above;
    const bool done = remaining == sh.count;  // every candidate left is kept
    __syncthreads();                          // sh.digit/above/count and the histograms are reused
    if (done) break;
  }
  // kept: (key & mask) > prefix, or (key & mask) == prefix among the first `remaining` by position
  const uint32_t kstar = prefix;
  const int need_eq = remaining;

  // ---- ordered write: tiles of kKeyCap positions, thread t owns kPer consecutive ones
  int eq_carry = 0, out_carry = 0;
  for (int b0 = 0; b0 < n; b0 += kKeyCap) {
    uint32_t key[kPer];
    int n_eq = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int j = b0 + tid * kPer + q;
      key[q] = j < n ? (key_at(j) & mask) : 0u;
      n_eq += (j < n && key[q] == kstar) ? 1 : 0;
    }
    int eq_tot;
    int eq_rank = eq_carry + block_incl_scan(n_eq, sh.wsum, &eq_tot) - n_eq;
    uint32_t keep_bits = 0;
    int n_keep = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int j = b0 + tid * kPer + q;
      bool kp = false;
      if (j < n) {
        if (key[q] > kstar) {
          kp = true;
        } else if (key[q] == kstar) {
          kp = eq_rank < need_eq;
          ++eq_rank;
        }
      }
      keep_bits |= (kp ? 1u : 0u) << q;
      n_keep += kp ? 1 : 0;
    }
    int keep_tot;
    int o = out_carry + block_incl_scan(n_keep, sh.wsum, &keep_tot) - n_keep;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      if ((keep_bits >> q) & 1u) kept_idx[base + o++] = static_cast<int32_t>(t0 + b0 + tid * kPer + q);
    }
    eq_carry += eq_tot;
    out_carry += keep_tot;
  }
}

// Candidates of the chosen first-pass bucket ranked directly, when there are at most this many.
constexpr int kCandCap = 256;

// Finishes the selection from the first-pass histogram when the image's keys are staged:
// the bucket holding the k-th largest key usually holds a few dozen keys, so they are
// gathered and ranked against each other (one compare per pair), which gives the k-th
// largest key thr directly. Then one block scan carries both the counts of keys above
// thr and of keys equal to it (16 bits each), and the kept positions are written in
// ascending order: every key above thr and the first k - #(key > thr) equal to it.
// Returns false (having written nothing) when the bucket is too large; all threads call.
// dry: compute everything but write nothing (warms the instruction cache).
__device__ __forceinline__ bool select_from_first_pass(int n, int k, int64_t t0, int64_t base,
                                                    int32_t* __restrict__ kept_idx, SelShared& sh, uint32_t kmin,
                                                    uint32_t kmax, bool dry) {
  const int tid = threadIdx.x;
  const int top = highest_differing_bit(kmin, kmax);
  const uint32_t mask = shared_bits_mask(top);
  const int shift = top >= 7 ? top - 7 : 0;
  const uint32_t dmask = (2u << (top - shift)) - 1u;
  choose_digit(sh, k);
  const int c1 = sh.count, remaining = k - sh.above;
  if (c1 > kCandCap) return false;
  const uint32_t bmask = mask | (dmask << shift);
  const uint32_t bval = (kmin & mask) | (static_cast<uint32_t>(sh.digit) << shift);
  uint32_t* cand = reinterpret_cast<uint32_t*>(&sh.hist[1][0]);  // the histograms are dead now
  for (int j = tid; j < n; j += kThreads) {
    const uint32_t key = sh.keys[j];
    if ((key & bmask) == bval) cand[atomicAdd(&sh.ncand, 1)] = key;
  }
  __syncthreads();
  if (tid < c1) {
    const uint32_t v = cand[tid];
    int gt = 0, ge = 0;
    for (int u = 0; u < c1; ++u) {
      const uint32_t w = cand[u];
      gt += w > v ? 1 : 0;
      ge += w >= v ? 1 : 0;
    }
    if (gt < remaining && remaining <= ge) sh.thr = v;
  }
  __syncthreads();
  const uint32_t thr = sh.thr;
  // thread t owns positions t*kPer .. t*kPer + kPer - 1
  const int j0 = tid * kPer;
  uint32_t kk[kPer];
  int gt = 0, eq = 0;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    kk[q] = j0 + q < n ? sh.keys[j0 + q] : 0u;
    gt += (j0 + q < n && kk[q] > thr) ? 1 : 0;
    eq += (j0 + q < n && kk[q] == thr) ? 1 : 0;
  }
  int tot;
  const int packed = gt | (eq << 16);
  const int pre = block_incl_scan(packed, sh.wsum, &tot) - packed;
  const int need_eq = k - (tot & 0xffff);
  int eq_rank = pre >> 16;
  int o = (pre & 0xffff) + min(eq_rank, need_eq);
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    if (j0 + q < n) {
      bool kp = kk[q] > thr;
      if (kk[q] == thr) kp = eq_rank++ < need_eq;
      if (kp && !dry) kept_idx[base + o] = static_cast<int32_t>(t0 + j0 + q);
      o += kp ? 1 : 0;
    }
  }
  return true;
}

// Stage the image's keys (when they fit) and find their range; all threads call.
__device__ void stage_and_range(const float* __restrict__ sc, int n, bool stage, SelShared& sh, uint32_t* kmin_out,
                                uint32_t* kmax_out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t lo = 0xffffffffu, hi = 0u;
  if (stage) {
    uint32_t v[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) {  // all loads in flight at once
      const int j = tid + q * kThreads;
      v[q] = j < n ? rank_key(sc[j]) : 0u;
    }
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int j = tid + q * kThreads;
      if (j < n) {
        sh.keys[j] = v[q];
        lo = min(lo, v[q]);
        hi = max(hi, v[q]);
      }
    }
  } else {
    for (int j = tid; j < n; j += kThreads) {
      const uint32_t key = rank_key(sc[j]);
      lo = min(lo, key);
      hi = max(hi, key);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(kFull, lo, o));
    hi = max(hi, __shfl_xor_sync(kFull, hi, o));
  }
  if (lane == 0) {
    sh.wmin[warp] = lo;
    sh.wmax[warp] = hi;
  }
  __syncthreads();
  lo = sh.wmin[0];
  hi = sh.wmax[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) {
    lo = min(lo, sh.wmin[w]);
    hi = max(hi, sh.wmax[w]);
  }
  *kmin_out = lo;
  *kmax_out = hi;
}

// Text before the first image of request r (the whole request if it has none).
__device__ void leading_text(const SelectArgs& a, int r) {
  const int Tr = a.cu[r + 1] - a.cu[r];
  const int first = (a.icu[r] < a.icu[r + 1]) ? a.ist[a.icu[r]] : Tr;
  const int64_t base = a.out_cu[r];
  if (base < 0 || base + first > a.out_cu[r + 1] || static_cast<int64_t>(a.out_cu[r + 1]) > a.n_kept) {
    if (threadIdx.x == 0) record_error(a.st, AVTP_ERR_DEVICE_INPUT, r);
    return;
  }
  for (int p = threadIdx.x; p < first; p += kThreads) a.kept_idx[base + p] = a.cu[r] + p;
}

__global__ void __launch_bounds__(kThreads)
k_select(SelectArgs a, const int32_t* __restrict__ budgets) {
  __shared__ SelShared sh;
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int b = blockIdx.x;
  if (b >= a.NI) {
    leading_text(a, b - a.NI);
    return;
  }
  const int i = b;
  const int r = a.img_req[i];
  const int i0 = a.icu[r], i1 = a.icu[r + 1];
  int before = 0, total = 0, bad = 0;
  for (int j = i0 + threadIdx.x; j < i1; j += kThreads) {
    const int kj = budgets[j];
    bad |= (kj < 0 || kj > a.iln[j]);
    total += kj;
    before += (j < i) ? kj : 0;
  }
  int sb, st, sbad;
  block_incl_scan(before, sh.wsum, &sb);
  block_incl_scan(total, sh.wsum, &st);
  block_incl_scan(bad, sh.wsum, &sbad);
  if (sbad) {
    if (threadIdx.x == 0) record_error(a.st, AVTP_ERR_DEVICE_INPUT, i);
    return;
  }
  const int Tr = a.cu[r + 1] - a.cu[r];
  const int ntxt = Tr - (a.vis_cu[i1] - a.vis_cu[i0]);
  if (a.out_cu[r] < 0 || a.out_cu[r + 1] - a.out_cu[r] != st + ntxt ||
      static_cast<int64_t>(a.out_cu[r + 1]) > a.n_kept) {
    if (threadIdx.x == 0) record_error(a.st, AVTP_ERR_DEVICE_INPUT, i);
    return;
  }
  const int s0 = a.ist[i], n = a.iln[i], k = budgets[i];
  const int64_t base = static_cast<int64_t>(a.out_cu[r]) + (s0 - (a.vis_cu[i] - a.vis_cu[i0])) + sb;
  const int64_t t0 = static_cast<int64_t>(a.cu[r]) + s0;
  const bool stage = n <= kKeyCap;
  uint32_t kmin, kmax;
  stage_and_range(a.scores + t0, n, stage, sh, &kmin, &kmax);
  block_select(a.scores + t0, n, k, t0, base, a.kept_idx, sh, stage, kmin, kmax, false);
  const int e = s0 + n;
  const int nxt = (i + 1 < i1) ? a.ist[i + 1] : Tr;
  for (int p = e + threadIdx.x; p < nxt; p += kThreads) a.kept_idx[base + k + (p - e)] = a.cu[r] + p;
}

struct AllocParams {
  const int64_t* img_sums;
  const float* keep_ratio;
  float alpha, r_min, r_max;
  int relative;
  int32_t* budgets;  // output: each CTA writes its own image's budget
  int m_cap;
  int warm_ctas;     // CTAs below this index warm their instruction cache before the wait
};

// What a CTA of k_alloc_select knows before the scores exist (from the call's inputs).
struct TailIn {
  int r, i0, m, li;
  int32_t s0, n, nxt, Tr;
  int64_t t0;
  // warp 0: the request's sizes and the scalars of the budget rule
  int32_t N, n_lane, vis_before;
  int64_t B, inv_n, inv_N;
  float kr;
  RatioRule rule;
};

// Keys of the CTA's image held per thread of warps 1..7 right after the wait.
constexpr int kTailKeys = (kKeyCap + kThreads - 33) / (kThreads - 32);

// Everything k_alloc_select does once the scores exist. The kernel runs it twice from one
// copy of the code (a loop that is not unrolled): first with dry set, before the wait, on
// whatever the buffers hold then (every index is in bounds for any contents; the sums are
// replaced by equal made-up means, so that the budget rule takes its common path),
// writing nothing to global memory; then for real. The dry run leaves exactly this code
// in the SM's instruction cache: a cold fetch costs about a microsecond per miss once the
// scoring stream has swept L2. Inlined, so that nothing of it lives on the stack (after
// the wait, local memory would come back from DRAM too).
// After the wait, one round of loads brings the status word, the request's sums, the
// request's output offsets and the image's scores, so that only one memory latency
// precedes the budget rule and the first histogram (which run side by side). The warm-up
// run loads the same way from shared memory (generic loads serve both): while the scores
// stream in, every global access waits behind them for microseconds.
__device__ __forceinline__ void alloc_select_tail(const SelectArgs& a, const AllocParams& ap, SelShared& sh,
                                                  const WarpAllocSmem& wsm, const WarpAllocSmem& wsm32,
                                                  const TailIn& in, bool dry) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.x;
  const int r = in.r, i0 = in.i0, m = in.m, li = in.li;
  const int32_t s0 = in.s0, nxt = in.nxt, Tr = in.Tr;
  const int32_t n = dry ? min(in.n, kKeyCap) : in.n;
  const int64_t t0 = in.t0;
  const bool image = b < a.NI;
  // where the loads below read: the call's buffers, or shared stand-ins for the warm-up
  const float* sc = dry ? reinterpret_cast<const float*>(sh.keys) : a.scores + t0;
  const int32_t* status = dry ? sh.dry_status : &a.st->layout_ok;
  const int64_t* sums = dry ? wsm32.S : ap.img_sums + i0;
  const int32_t* out_cu = dry ? sh.dry_out : a.out_cu + r;
  const bool stage = n <= kKeyCap;

  // ---- one round of loads
  const int layout_ok = *status;
  int64_t S_lane = 0;
  int32_t out_lo = 0, out_hi = 0;
  uint32_t key[kTailKeys];
  if (warp == 0) {
    if (image && lane < m && m <= 32) S_lane = sums[lane];
    if (image) {
      out_lo = out_cu[0];
      out_hi = out_cu[1];
    }
  } else if (image && stage) {
    const int wt = tid - 32;
#pragma unroll
    for (int q = 0; q < kTailKeys; ++q) {
      const int j = wt + q * (kThreads - 32);
      key[q] = j < n ? rank_key(sc[j]) : 0u;
    }
  }
  if (dry) S_lane = lane < m ? (static_cast<int64_t>(in.n_lane) << 30) : 0;  // equal means
  if (!layout_ok) return;
  if (!image) {
    if (!dry) leading_text(a, b - a.NI);
    return;
  }
  const int i = b;
  if (warp == 0) {
    // ---- the budget rule, one warp
    int err;
    int k, before, total;
    if (m <= 32) {
#ifdef AVTP_TIMELINE
      if (!dry && __shfl_sync(kFull, S_lane, 0) != INT64_MIN && lane == 0) timeline_stamp(a.st, kTlRuleBegin);
#endif
      int32_t K;
      err = warp_allocate32(wsm32, m, S_lane, in.n_lane, in.inv_n, in.B, in.N, in.inv_N, in.rule, ap.alpha, ap.r_min,
                            ap.r_max, &K);
      k = __shfl_sync(kFull, K, li);
      before = static_cast<int>(__reduce_add_sync(kFull, static_cast<uint32_t>(lane < li ? K : 0)));
      total = static_cast<int>(__reduce_add_sync(kFull, static_cast<uint32_t>(lane < m ? K : 0)));
    } else {
      for (int j = lane; j < m; j += 32) wsm.S[j] = dry ? (static_cast<int64_t>(wsm.n[j]) << 30) : ap.img_sums[i0 + j];
      __syncwarp();
      err = warp_allocate(wsm, m, in.B, in.N, in.kr, ap.alpha, ap.r_min, ap.r_max, ap.relative);
      int bs = 0, ts = 0;
      for (int j = lane; j < m; j += 32) {
        ts += wsm.K[j];
        bs += j < li ? wsm.K[j] : 0;
      }
      before = warp_sum(bs);
      total = warp_sum(ts);
      k = wsm.K[li];
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) sh.hist[0][lane * 8 + q] = 0;  // warp 0 takes no part in the first pass
    if (lane == 0) {
      if (!dry) timeline_stamp(a.st, kTlRuleEnd);
      sh.k = k;
      sh.before = before;
      sh.total = total;
      sh.alloc_err = err;
      sh.out_lo = out_lo;
      sh.out_hi = out_hi;
      sh.vis_before = in.vis_before;
      sh.n_vis = in.N;
    }
  } else {
    // ---- warps 1..7: stage the keys, find their range, build the first histogram
    const int wt = tid - 32;
    uint32_t lo = 0xffffffffu, hi = 0u;
    if (stage) {
#pragma unroll
      for (int q = 0; q < kTailKeys; ++q) {
        const int j = wt + q * (kThreads - 32);
        if (j < n) {
          sh.keys[j] = key[q];
          lo = min(lo, key[q]);
          hi = max(hi, key[q]);
        }
      }
    } else {
      for (int j = wt; j < n; j += kThreads - 32) {
        const uint32_t kk = rank_key(sc[j]);
        lo = min(lo, kk);
        hi = max(hi, kk);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = min(lo, __shfl_xor_sync(kFull, lo, o));
      hi = max(hi, __shfl_xor_sync(kFull, hi, o));
    }
    if (lane == 0) {
      sh.wmin[warp] = lo;
      sh.wmax[warp] = hi;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) sh.hist[warp][lane * 8 + q] = 0;
    bar_workers();  // ranges published, keys staged, sub-histograms cleared
    lo = sh.wmin[1];
    hi = sh.wmax[1];
#pragma unroll
    for (int w = 2; w < kWarps; ++w) {
      lo = min(lo, sh.wmin[w]);
      hi = max(hi, sh.wmax[w]);
    }
    const int top = highest_differing_bit(lo, hi);
    if (top >= 0) {
      const uint32_t mask = shared_bits_mask(top);
      const int shift = top >= 7 ? top - 7 : 0;
      const uint32_t dmask = (2u << (top - shift)) - 1u;
      hist_pass(KeySource{sc, stage ? sh.keys : nullptr}, n, mask, lo & mask, shift, dmask, sh.hist[warp], wt,
                kThreads - 32);
    }
#ifdef AVTP_TIMELINE
    bar_workers();  // every worker's first pass is done
    if (!dry && tid == 32) timeline_stamp(a.st, kTlHistDone);
#endif
    if (tid == 32) {
      sh.kmin = lo;
      sh.kmax = hi;
      sh.ncand = 0;
    }
  }
  __syncthreads();
  const uint32_t kmin = sh.kmin, kmax = sh.kmax;
  const int k = sh.k, before = sh.before, total = sh.total;
  const int32_t olo = sh.out_lo, ohi = sh.out_hi, vis_b = sh.vis_before, Nv = sh.n_vis;
  if (!dry) {
    if (sh.alloc_err != AVTP_OK) {
      if (tid == 0) record_error(a.st, sh.alloc_err, r);
      return;
    }
    if (tid == 0) ap.budgets[i] = k;
    if (olo < 0 || ohi - olo != total + (Tr - Nv) || static_cast<int64_t>(ohi) > a.n_kept) {
      if (tid == 0) record_error(a.st, AVTP_ERR_DEVICE_INPUT, i);
      return;
    }
  }
  const int64_t base = static_cast<int64_t>(olo) + (s0 - vis_b) + before;
  const bool fast = stage && kmin != kmax && k > 0 && k < n &&
                    select_from_first_pass(n, k, t0, base, a.kept_idx, sh, kmin, kmax, dry);
  if (dry) {
    __syncthreads();  // the shared state is reused by the real run
    return;
  }
  if (!fast) block_select(sc, n, k, t0, base, a.kept_idx, sh, stage, kmin, kmax, kmin != kmax);
  const int e = s0 + n;
  for (int p = e + tid; p < nxt; p += kThreads) a.kept_idx[base + k + (p - e)] = a.cu[r] + p;
  if (tid == 0) timeline_stamp(a.st, kTlSelEnd);
}

// 184 registers: the tail runs without spilling (at 128 it spilled about 100 bytes a
// thread, and local memory is slow to come back right after the scoring stream). One CTA
// per SM, which is how the free SMs are used anyway.
__global__ void __maxnreg__(184)
k_alloc_select(SelectArgs a, AllocParams ap) {
  extern __shared__ __align__(16) unsigned char dsmem[];  // budget scratch for requests of > 32 images
  __shared__ __align__(16) unsigned char rule32[warp_alloc_smem_bytes(32)];  // ... and of at most 32
  __shared__ SelShared sh;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.x;
  if (tid == 0) timeline_stamp(a.st, kTlSelBegin);
  const WarpAllocSmem wsm = carve_warp_alloc(dsmem, ap.m_cap);
  const WarpAllocSmem wsm32 = carve_warp_alloc(rule32, 32);

  // ---- set-up from the call's inputs only, overlapped with the scoring kernel.
  // The layout is not validated yet, so every index is clamped; nothing here is
  // used unless the validation kernel accepts the layout.
  TailIn in{};
  if (b < a.NI) {
    in.r = upper_index(a.icu, a.R, b);
    in.i0 = min(max(a.icu[in.r], 0), a.NI);
    const int i1 = min(max(a.icu[in.r + 1], in.i0), a.NI);
    in.m = min(i1 - in.i0, ap.m_cap);
    if (in.m > 0) {
      in.li = min(max(b - in.i0, 0), in.m - 1);
      in.Tr = a.cu[in.r + 1] - a.cu[in.r];
      in.s0 = a.ist[in.i0 + in.li];
      in.n = a.iln[in.i0 + in.li];
      in.nxt = (in.li + 1 < in.m) ? a.ist[in.i0 + in.li + 1] : in.Tr;
      in.t0 = static_cast<int64_t>(a.cu[in.r]) + in.s0;
    }
    // a span outside the scores (a malformed layout, reported by the validation kernel)
    // is never read, not even by the dry run
    if (in.t0 < 0 || in.n < 0 || in.t0 + in.n > a.T) {
      in.t0 = 0;
      in.n = 0;
    }
  }
  if (warp == 0 && b < a.NI) {
    int64_t nsum = 0, nbefore = 0;
    for (int j = lane; j < in.m; j += 32) {
      const int32_t nj = a.iln[in.i0 + j];
      if (in.m > 32) wsm.n[j] = nj;
      else in.n_lane = nj;
      nsum += nj;
      nbefore += j < in.li ? nj : 0;
    }
    in.N = static_cast<int32_t>(warp_sum(nsum));
    in.vis_before = static_cast<int32_t>(warp_sum(nbefore));
    in.kr = ap.keep_ratio[in.r];
    // B_r = floor(r_base * N_vis + 0.5), each operation rounded once
    in.B = static_cast<int64_t>(
        floor(__dadd_rn(__dmul_rn(static_cast<double>(in.kr), static_cast<double>(in.N)), 0.5)));
    in.rule = make_ratio_rule(in.kr, ap.alpha, ap.relative);
    in.inv_N = recip62(in.N);
    in.inv_n = recip62(in.n_lane);
  }

  if (tid == 0) {
    sh.dry_status[0] = sh.dry_status[1] = sh.dry_status[2] = sh.dry_status[3] = 1;
    sh.dry_out[0] = 0;
    sh.dry_out[1] = 0;
  }
  __syncthreads();
  // ---- the dry run (see alloc_select_tail) on the CTAs that start while the scores
  // stream in (prune_reserve_sms), then the wait for the scores and per-image sums (and,
  // through them, the validation), then the real run: one copy of the code for both
#pragma unroll 1
  for (int pass = b < ap.warm_ctas ? 0 : 1; pass < 2; ++pass) {
    if (pass == 1) {
      if (tid == 0 && b < ap.warm_ctas) timeline_stamp(a.st, kTlSelDryEnd);
      pdl_wait();
      pdl_trigger();
      if (tid == 0) timeline_stamp(a.st, kTlSelWaited);
    }
    alloc_select_tail(a, ap, sh, wsm, wsm32, in, pass == 0);
  }
}

SelectArgs make_args(const avtp_layout_t& L, const float* scores, const int32_t* out_cu_seqlens, int32_t* kept_idx,
                     int64_t n_kept, void* ws, const WsPlan& p) {
  SelectArgs a;
  a.cu = L.cu_seqlens;
  a.icu = L.img_cu;
  a.ist = L.img_start;
  a.iln = L.img_len;
  a.R = L.n_requests;
  a.NI = L.n_images;
  a.T = L.n_tokens;
  a.scores = scores;
  a.out_cu = out_cu_seqlens;
  a.kept_idx = kept_idx;
  a.n_kept = n_kept;
  a.vis_cu = ws_at<int32_t>(ws, p.vis_cu);
  a.img_req = ws_at<int32_t>(ws, p.img_req);
  a.st = ws_at<DevStatus>(ws, p.status);
  return a;
}

}  // namespace

cudaError_t launch_select(const avtp_layout_t& L, const float* scores, const int32_t* budgets,
                          const int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, void* ws,
                          const WsPlan& p, cudaStream_t s) {
  const SelectArgs a = make_args(L, scores, out_cu_seqlens, kept_idx, n_kept, ws, p);
  return launch_kernel(k_select, dim3(L.n_images + L.n_requests), dim3(kThreads), 0, s, /*pdl=*/true, a, budgets);
}

cudaError_t launch_alloc_select(const avtp_layout_t& L, const int64_t* img_sums, const avtp_alloc_args_t& aa,
                                int32_t* budgets, const float* scores, const int32_t* out_cu_seqlens,
                                int32_t* kept_idx, int64_t n_kept, void* ws, const WsPlan& p, cudaStream_t s,
                                int warm_ctas) {
  const SelectArgs a = make_args(L, scores, out_cu_seqlens, kept_idx, n_kept, ws, p);
  AllocParams ap;
  ap.img_sums = img_sums;
  ap.keep_ratio = aa.keep_ratio;
  ap.alpha = aa.alpha;
  ap.r_min = aa.r_min;
  ap.r_max = aa.r_max;
  ap.relative = aa.relative;
  ap.budgets = budgets;
  ap.warm_ctas = warm_ctas;
  ap.m_cap = L.n_images < kMaxImagesPerRequest ? L.n_images : kMaxImagesPerRequest;
  if (ap.m_cap < 1) ap.m_cap = 1;
  // the budget scratch is only used for requests of more than 32 images
  const size_t smem = ap.m_cap > 32 ? warp_alloc_smem_bytes(ap.m_cap) : 0;
  // same shared-memory configuration as the scoring kernels, so that a CTA of this
  // kernel can start on an SM where a scoring CTA still runs
  static PerDevice carveout;
  const cudaError_t ce = once_per_device(carveout, [](int, int*) {
    return cudaFuncSetAttribute(k_alloc_select, cudaFuncAttributePreferredSharedMemoryCarveout,
                                cudaSharedmemCarveoutMaxShared);
  });
  if (ce != cudaSuccess) return ce;
  if (smem > 16 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_alloc_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  return launch_kernel(k_alloc_select, dim3(L.n_images + L.n_requests), dim3(kThreads), smem, s, /*pdl=*/true, a,
                       ap);
}

}  // namespace avtp
