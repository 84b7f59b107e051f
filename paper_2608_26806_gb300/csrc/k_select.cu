// Step 3: per-image top-k, text always kept, positions emitted in ascending order
// (paper §3.1: the pruned sequence is an order-preserving subsequence; §3.3.3:
// image i keeps its k_i most important tokens).
//
// One CTA per image, plus one CTA per request for the text before its first image.
// Ranking: order-preserving 32-bit keys (score descending; NaN lowest; -0 == +0),
// ties by lower position. A 4-pass 8-bit radix select finds the k-th key K*;
// tokens above K* are kept, and of those equal to K* the first (by position)
// k - #{key > K*}. Kept positions are written in order with block-wide scans.
// The CTA also writes the text run that follows its image.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kItems = 4;
constexpr int kTile = kThreads * kItems;

// Exclusive block scan of one int per thread; returns the block total via *total.
__device__ __forceinline__ int block_excl_scan(int v, int* s_warp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  int pre = 0, tot = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    const int t = s_warp[w];
    pre += (w < warp) ? t : 0;
    tot += t;
  }
  *total = tot;
  return pre + x - v;
}

__device__ __forceinline__ int block_sum_int(int v, int* s_warp) {
  int tot;
  block_excl_scan(v, s_warp, &tot);
  return tot;
}

__global__ void __launch_bounds__(kThreads)
k_select(const int32_t* __restrict__ cu, const int32_t* __restrict__ icu, const int32_t* __restrict__ ist,
         const int32_t* __restrict__ iln, int R, int NI, const float* __restrict__ scores,
         const int32_t* __restrict__ budgets, const int32_t* __restrict__ out_cu, int32_t* __restrict__ kept_idx,
         int64_t n_kept, const int32_t* __restrict__ vis_cu, const int32_t* __restrict__ img_req, DevStatus* st) {
  __shared__ int s_hist[256];
  __shared__ int s_warp[kWarps];
  __shared__ int s_digit, s_above;
  if (!st->layout_ok) return;
  const int tid = threadIdx.x;
  const int b = blockIdx.x;

  if (b >= NI) {  // text before the first image of request r (the whole request if it has none)
    const int r = b - NI;
    const int Tr = cu[r + 1] - cu[r];
    const int first = (icu[r] < icu[r + 1]) ? ist[icu[r]] : Tr;
    const int64_t base = out_cu[r];
    if (base < 0 || base + first > out_cu[r + 1] || static_cast<int64_t>(out_cu[r + 1]) > n_kept) {
      if (tid == 0) record_error(st, AVTP_ERR_DEVICE_INPUT, r);
      return;
    }
    for (int p = tid; p < first; p += kThreads) kept_idx[base + p] = cu[r] + p;
    return;
  }

  const int i = b;
  const int r = img_req[i];
  const int i0 = icu[r], i1 = icu[r + 1];
  // kept tokens of earlier images of this request, and the request's total; validate budgets
  int before = 0, total = 0, bad = 0;
  for (int j = i0 + tid; j < i1; j += kThreads) {
    const int kj = budgets[j];
    bad |= (kj < 0 || kj > iln[j]);
    total += kj;
    before += (j < i) ? kj : 0;
  }
  before = block_sum_int(before, s_warp);
  total = block_sum_int(total, s_warp);
  bad = block_sum_int(bad, s_warp);
  const int Tr = cu[r + 1] - cu[r];
  const int ntxt = Tr - (vis_cu[i1] - vis_cu[i0]);
  if (bad || out_cu[r] < 0 || out_cu[r + 1] - out_cu[r] != total + ntxt ||
      static_cast<int64_t>(out_cu[r + 1]) > n_kept) {
    if (tid == 0) record_error(st, AVTP_ERR_DEVICE_INPUT, i);
    return;
  }
  const int s0 = ist[i], n = iln[i], k = budgets[i];
  const int64_t base = static_cast<int64_t>(out_cu[r]) + (s0 - (vis_cu[i] - vis_cu[i0])) + before;
  const int64_t t0 = static_cast<int64_t>(cu[r]) + s0;  // packed position of the image's first token
  const float* sc = scores + t0;

  if (k == n) {
    for (int j = tid; j < n; j += kThreads) kept_idx[base + j] = static_cast<int32_t>(t0 + j);
  } else if (k > 0) {
    // ---- radix select of the k-th largest key
    uint32_t prefix = 0, mask = 0;
    int remaining = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
      s_hist[tid] = 0;  // kThreads == 256 bins
      __syncthreads();
      for (int base_j = 0; base_j < n; base_j += kTile) {
#pragma unroll
        for (int it = 0; it < kItems; ++it) {
          const int j = base_j + tid * kItems + it;
          if (j < n) {
            const uint32_t key = rank_key(sc[j]);
            if ((key & mask) == prefix) atomicAdd(&s_hist[(key >> shift) & 255u], 1);
          }
        }
      }
      __syncthreads();
      // thread t looks at digit 255 - t; inclusive prefix = count with digit >= 255 - t
      const int c = s_hist[255 - tid];
      int tot;
      const int excl = block_excl_scan(c, s_warp, &tot);
      if (excl < remaining && remaining <= excl + c) {
        s_digit = 255 - tid;
        s_above = excl;
      }
      __syncthreads();
      prefix |= static_cast<uint32_t>(s_digit) << shift;
      mask |= 0xFFu << shift;
      remaining -= s_above;
      __syncthreads();
    }
    const uint32_t kstar = prefix;
    const int need_eq = remaining;  // tokens equal to K* to keep, lowest positions first
    // ---- ordered write
    int eq_carry = 0, out_carry = 0;
    for (int base_j = 0; base_j < n; base_j += kTile) {
      uint32_t key[kItems];
      int n_eq = 0;
#pragma unroll
      for (int it = 0; it < kItems; ++it) {
        const int j = base_j + tid * kItems + it;
        key[it] = (j < n) ? rank_key(sc[j]) : 0u;
        n_eq += (j < n && key[it] == kstar) ? 1 : 0;
      }
      int eq_tot;
      int eq_rank = eq_carry + block_excl_scan(n_eq, s_warp, &eq_tot);
      bool keep[kItems];
      int n_keep = 0;
#pragma unroll
      for (int it = 0; it < kItems; ++it) {
        const int j = base_j + tid * kItems + it;
        bool kp = false;
        if (j < n) {
          if (key[it] > kstar) kp = true;
          else if (key[it] == kstar) { kp = eq_rank < need_eq; ++eq_rank; }
        }
        keep[it] = kp;
        n_keep += kp ? 1 : 0;
      }
      int keep_tot;
      int o = out_carry + block_excl_scan(n_keep, s_warp, &keep_tot);
#pragma unroll
      for (int it = 0; it < kItems; ++it) {
        const int j = base_j + tid * kItems + it;
        if (keep[it]) kept_idx[base + o++] = static_cast<int32_t>(t0 + j);
      }
      eq_carry += eq_tot;
      out_carry += keep_tot;
    }
  }

  // ---- the text run after this image
  const int e = s0 + n;
  const int nxt = (i + 1 < i1) ? ist[i + 1] : Tr;
  for (int p = e + tid; p < nxt; p += kThreads) kept_idx[base + k + (p - e)] = cu[r] + p;
}

}  // namespace

cudaError_t launch_select(const avtp_layout_t& L, const float* scores, const int32_t* budgets,
                          const int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, void* ws,
                          const WsPlan& p, cudaStream_t s) {
  const int grid = L.n_images + L.n_requests;
  k_select<<<grid, kThreads, 0, s>>>(L.cu_seqlens, L.img_cu, L.img_start, L.img_len, L.n_requests, L.n_images, scores,
                                      budgets, out_cu_seqlens, kept_idx, n_kept, ws_at<int32_t>(ws, p.vis_cu),
                                      ws_at<int32_t>(ws, p.img_req), ws_at<DevStatus>(ws, p.status));
  return cudaGetLastError();
}

}  // namespace avtp
