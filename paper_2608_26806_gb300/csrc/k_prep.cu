// Layout validation and per-call bookkeeping, run once at the start of every
// entry point that reads the layout. One CTA: the layout arrays are small
// (requests and images, not tokens), except the optional text index list.
//
// Writes into the workspace: the status word, vis_cu (visual-token prefix over
// all images), img_req (request of each image), and optionally the global
// budgets B_r = floor(r_base * N_vis + 0.5) (paper §3.3.3 base keep ratio),
// out_cu_seqlens, the text-query bookkeeping of the attention criterion, and the
// image spans of the pruned batch (progressive pruning, paper §3.3.2).
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kPrepThreads = 1024;

// Block-wide exclusive scan of value(i), i in [0, n): out[i] = sum_{j<i}, out[n] = total.
template <typename T, typename F>
__device__ T block_exclusive_scan(int n, F value, T* out, T* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  T carry = 0;
  for (int base = 0; base < n; base += blockDim.x) {
    const int i = base + threadIdx.x;
    const T v = (i < n) ? value(i) : T(0);
    T x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      T y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
      T w = (lane < nwarps) ? s_warp[lane] : T(0);
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        T y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      s_warp[lane] = w;
    }
    __syncthreads();
    const T warp_prefix = (warp > 0) ? s_warp[warp - 1] : T(0);
    if (i < n) out[i] = carry + warp_prefix + x - v;
    const T chunk_total = s_warp[nwarps - 1];
    __syncthreads();
    carry += chunk_total;
  }
  if (threadIdx.x == 0) out[n] = carry;
  __syncthreads();
  return carry;
}

// Layout arrays are staged in shared memory when they fit. Kept small (10 KiB) so
// that this one-CTA kernel can share an SM with a CTA of the scoring kernel,
// which is launched while this kernel still runs.
constexpr int kStageInts = 2560;

__global__ void __launch_bounds__(kPrepThreads)
k_prep(PrepArgs a, DevStatus* st, int32_t* g_vis_cu, int32_t* g_img_req, int32_t* req_budget, int32_t* text_idx,
       int32_t* text_cu, int32_t* blk_cu, int32_t* p1s_cu, int32_t* p2t_cu, int32_t* ktile_cu, int32_t* ktile_img,
       int32_t* meta, int32_t* g_scratch) {
  __shared__ int s_err, s_detail, s_max_steps;
  __shared__ int32_t s_warp[32];
  __shared__ int32_t s_stage[kStageInts];
  // The first kernel of a call: it is launched after everything before it in the
  // stream has finished, so the next kernel may be scheduled at once.
  pdl_trigger();
  const int tid = threadIdx.x;
  if (tid == 0) timeline_stamp(st, kTlPrepBegin);
  const int R = a.L.n_requests, NI = a.L.n_images;
  const int64_t T = a.L.n_tokens;
  const int32_t* cu = a.L.cu_seqlens;
  const int32_t* icu = a.L.img_cu;
  const int32_t* ist = a.L.img_start;
  const int32_t* iln = a.L.img_len;
  int32_t* vis_cu = g_vis_cu;
  int32_t* img_req = g_img_req;
  // Stage the small layout arrays in shared memory: one round trip to global
  // memory instead of one per dependent step below.
  const bool staged = 2 * static_cast<int64_t>(R) + 4 * static_cast<int64_t>(NI) + 3 <= kStageInts;
  if (staged) {
    int32_t* s_cu = s_stage;
    int32_t* s_icu = s_cu + (R + 1);
    int32_t* s_ist = s_icu + (R + 1);
    int32_t* s_iln = s_ist + NI;
    int32_t* s_vis = s_iln + NI;
    int32_t* s_req = s_vis + (NI + 1);
    for (int j = tid; j <= R; j += blockDim.x) {
      s_cu[j] = cu[j];
      s_icu[j] = icu[j];
    }
    for (int j = tid; j < NI; j += blockDim.x) {
      s_ist[j] = ist[j];
      s_iln[j] = iln[j];
    }
    cu = s_cu;
    icu = s_icu;
    ist = s_ist;
    iln = s_iln;
    vis_cu = s_vis;
    img_req = s_req;
  }
  if (tid == 0) { s_err = 0; s_detail = -1; }
  __syncthreads();
  auto fail = [&](int code, int detail) {
    if (atomicCAS(&s_err, 0, code) == 0) s_detail = detail;
  };

  // Phase 0: offsets arrays.
  if (tid == 0) {
    if (cu[0] != 0 || static_cast<int64_t>(cu[R]) != T || icu[0] != 0 || icu[R] != NI) fail(AVTP_ERR_DEVICE_INPUT, -1);
  }
  for (int r = tid; r < R; r += blockDim.x) {
    if (cu[r + 1] < cu[r] || icu[r + 1] < icu[r]) fail(AVTP_ERR_DEVICE_INPUT, r);
    else if (icu[r + 1] - icu[r] > kMaxImagesPerRequest) fail(AVTP_ERR_RANGE, r);
  }
  __syncthreads();

  // Phase 1: image spans (inside their request, >= 1 token, sorted, disjoint).
  if (s_err == 0) {
    for (int i = tid; i < NI; i += blockDim.x) {
      const int r = upper_index(icu, R, i);
      const int64_t Tr = static_cast<int64_t>(cu[r + 1]) - cu[r];
      const int64_t s0 = ist[i], n0 = iln[i];
      bool bad = n0 < 1 || s0 < 0 || s0 + n0 > Tr;
      if (!bad && i > icu[r]) bad = s0 < static_cast<int64_t>(ist[i - 1]) + iln[i - 1];
      if (bad) fail(AVTP_ERR_DEVICE_INPUT, i);
      img_req[i] = r;
    }
  }
  __syncthreads();

  if (s_err == 0) {
    // Phase 2: visual prefix over all images.
    block_exclusive_scan<int32_t>(NI, [&](int i) { return iln[i]; }, vis_cu, s_warp);
    for (int r = tid; r < R; r += blockDim.x) {
      if (vis_cu[icu[r + 1]] - vis_cu[icu[r]] > kMaxVisualPerRequest) fail(AVTP_ERR_RANGE, r);
    }
    __syncthreads();
  }

  if (s_err == 0 && a.keep_ratio != nullptr) {
    // Phase 3: global budgets B_r and the packed offsets of the pruned batch.
    for (int r = tid; r < R; r += blockDim.x) {
      const float kr = a.keep_ratio[r];
      const int32_t nvis = vis_cu[icu[r + 1]] - vis_cu[icu[r]];
      if (!(kr >= a.r_min && kr <= a.r_max) || !multiple_of_2m32(kr)) {
        fail(AVTP_ERR_DEVICE_INPUT, r);
        req_budget[r] = 0;
      } else {
        const double x = __dadd_rn(__dmul_rn(static_cast<double>(kr), static_cast<double>(nvis)), 0.5);
        req_budget[r] = static_cast<int32_t>(floor(x));
      }
    }
    __syncthreads();
    if (a.out_cu_seqlens != nullptr) {
      block_exclusive_scan<int32_t>(
          R,
          [&](int r) {
            const int32_t nvis = vis_cu[icu[r + 1]] - vis_cu[icu[r]];
            return req_budget[r] + (cu[r + 1] - cu[r] - nvis);
          },
          a.out_cu_seqlens, s_warp);
    }
  }

  if (s_err == 0 && a.build_text_tiles) {
    // Phase 4: text ordinals. Text ordinal of packed token t = t - (visual tokens before t).
    for (int r = tid; r <= R; r += blockDim.x) text_cu[r] = cu[r] - vis_cu[icu[r]];
    __syncthreads();
    const int lane = tid & 31, warp = tid >> 5, nwarps = blockDim.x >> 5;
    for (int run = warp; run < NI + R; run += nwarps) {
      int r, p0, p1, base;
      if (run < NI) {  // text after image `run`, up to the next image or the request end
        const int i = run;
        r = img_req[i];
        const int Tr = cu[r + 1] - cu[r];
        p0 = ist[i] + iln[i];
        p1 = (i + 1 < icu[r + 1]) ? ist[i + 1] : Tr;
        base = text_cu[r] + p0 - (vis_cu[i + 1] - vis_cu[icu[r]]);
      } else {  // text before the first image of request r
        r = run - NI;
        const int Tr = cu[r + 1] - cu[r];
        p0 = 0;
        p1 = (icu[r] < icu[r + 1]) ? ist[icu[r]] : Tr;
        base = text_cu[r];
      }
      for (int p = p0 + lane; p < p1; p += 32) text_idx[base + (p - p0)] = cu[r] + p;
    }
    __syncthreads();
    const int G = a.attn.G;
    if (tid == 0 && static_cast<int64_t>(text_cu[R]) > a.attn.max_text) fail(AVTP_ERR_RANGE, -1);
    __syncthreads();
    if (s_err == 0) {
      // Row blocks of kAttnBlockRows (text query, head) rows per request.
      block_exclusive_scan<int32_t>(
          R, [&](int r) { return ((text_cu[r + 1] - text_cu[r]) * G + kAttnBlockRows - 1) / kAttnBlockRows; }, blk_cu,
          s_warp);
      const int NB = blk_cu[R];
      // Key tiles of kAttnTileM visual keys per image.
      block_exclusive_scan<int32_t>(
          NI, [&](int i) { return (iln[i] + kAttnTileM - 1) / kAttnTileM; }, ktile_cu, s_warp);
      for (int i = tid; i < NI; i += blockDim.x)
        for (int t = ktile_cu[i]; t < ktile_cu[i + 1]; ++t) ktile_img[t] = i;
      // Pass 2 of block b: the key tiles of every image that at least one of the block's
      // queries follows. Images are sorted and the text ordinal of the first token after
      // image i, o_first(i), does not decrease with i, so those images are a prefix.
      auto p2_tiles = [&](int b) {
        const int r = upper_index(blk_cu, R, b);
        const int64_t R0 = static_cast<int64_t>(text_cu[r]) * G + static_cast<int64_t>(b - blk_cu[r]) * kAttnBlockRows;
        const int64_t R1 = min(R0 + kAttnBlockRows, static_cast<int64_t>(text_cu[r + 1]) * G);
        int lo = icu[r], hi = icu[r + 1];  // first image in [lo, hi) with o_first * G >= R1
        while (lo < hi) {
          const int i = (lo + hi) >> 1;
          const int64_t o_first =
              static_cast<int64_t>(text_cu[r]) + ist[i] + iln[i] - (vis_cu[i + 1] - vis_cu[icu[r]]);
          if (o_first * G >= R1) hi = i; else lo = i + 1;
        }
        return ktile_cu[lo] - ktile_cu[icu[r]];
      };
      block_exclusive_scan<int32_t>(NB, p2_tiles, p2t_cu, s_warp);
      // Pass 1 of block b: steps of kAttnTileN keys from the request's first token to its
      // last query (none when pass 2 has nothing for the block).
      if (tid == 0) s_max_steps = 0;
      __syncthreads();
      auto p1_steps = [&](int b) {
        if (p2t_cu[b + 1] == p2t_cu[b]) return 0;
        const int r = upper_index(blk_cu, R, b);
        const int64_t R0 = static_cast<int64_t>(text_cu[r]) * G + static_cast<int64_t>(b - blk_cu[r]) * kAttnBlockRows;
        const int64_t R1 = min(R0 + kAttnBlockRows, static_cast<int64_t>(text_cu[r + 1]) * G);
        const int keys = text_idx[(R1 - 1) / G] - cu[r] + 1;
        const int steps = (keys + kAttnTileN - 1) / kAttnTileN;
        atomicMax(&s_max_steps, steps);
        return steps;
      };
      block_exclusive_scan<int32_t>(NB, p1_steps, p1s_cu, s_warp);
      if (tid == 0) {
        // Each CTA of a persistent pass takes a contiguous run of C steps of the flat
        // list (KV group, block, step). C1 also keeps a row's pass-1 partials within
        // kAttnMaxChunks slots: a block of S steps meets at most (S - 1) / C1 + 2 CTAs.
        const int64_t grid = a.attn.grid > 0 ? a.attn.grid : 1;
        const int64_t F1 = p1s_cu[NB], F2 = p2t_cu[NB];
        int64_t C1 = (a.attn.Hkv * F1 + grid - 1) / grid;
        const int64_t c_min = (s_max_steps - 1 + kAttnMaxChunks - 3) / (kAttnMaxChunks - 2);
        C1 = max(max(C1, c_min), static_cast<int64_t>(1));
        const int64_t C2 = max((a.attn.Hkv * F2 + grid - 1) / grid, static_cast<int64_t>(1));
        meta[0] = static_cast<int32_t>(F1);
        meta[1] = static_cast<int32_t>(C1);
        meta[2] = static_cast<int32_t>(F2);
        meta[3] = static_cast<int32_t>(C2);
      }
    }
  }

  if (s_err == 0 && a.zero_img_sums != nullptr) {
    for (int i = tid; i < NI; i += blockDim.x) a.zero_img_sums[i] = 0;
  }
  __syncthreads();
  if (staged && s_err == 0) {
    for (int j = tid; j <= NI; j += blockDim.x) g_vis_cu[j] = vis_cu[j];
    for (int j = tid; j < NI; j += blockDim.x) g_img_req[j] = img_req[j];
  }
  if (tid == 0) {
    st->code = s_err;
    st->detail = s_detail;
    st->pool = 0;
    st->layout_ok = (s_err == 0) ? 1 : 0;
    timeline_stamp(st, kTlPrepEnd);
  }
  if (a.pl_budgets != nullptr) {
    // The image spans of the pruned batch: image i of request r moves left by the tokens
    // pruned from the request's earlier images and keeps budgets[i] tokens (an exclusive
    // scan of the pruned counts over all images, less the request's first entry). A budget
    // outside [0, img_len] is recorded (after the status word above is written) and its
    // image gets an empty span.
    __syncthreads();
    if (s_err == 0) {
      const int32_t* budgets = a.pl_budgets;
      block_exclusive_scan<int32_t>(
          NI,
          [&](int i) {
            const int32_t k = budgets[i], n = iln[i];
            return (k >= 0 && k <= n) ? n - k : 0;
          },
          g_scratch, s_warp);
      for (int i = tid; i < NI; i += blockDim.x) {
        const int32_t k = budgets[i], n = iln[i];
        if (k < 0 || k > n) {
          record_error(st, AVTP_ERR_DEVICE_INPUT, i);
          a.pl_out_start[i] = 0;
          a.pl_out_len[i] = 0;
          continue;
        }
        const int first = icu[img_req[i]];  // the request's first image
        a.pl_out_start[i] = ist[i] - (g_scratch[i] - g_scratch[first]);
        a.pl_out_len[i] = k;
      }
    }
  }
}

}  // namespace

cudaError_t launch_prep(const PrepArgs& a, void* ws, const WsPlan& p, cudaStream_t s) {
  const bool b = a.build_text_tiles != 0;
  k_prep<<<1, kPrepThreads, 0, s>>>(a, ws_at<DevStatus>(ws, p.status), ws_at<int32_t>(ws, p.vis_cu),
                                    ws_at<int32_t>(ws, p.img_req), ws_at<int32_t>(ws, p.req_budget),
                                    b ? ws_at<int32_t>(ws, p.text_idx) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.text_cu) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.blk_cu) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.p1s_cu) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.p2t_cu) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.ktile_cu) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.ktile_img) : nullptr,
                                    b ? ws_at<int32_t>(ws, p.meta) : nullptr,
                                    a.pl_budgets != nullptr ? ws_at<int32_t>(ws, p.scratch) : nullptr);
  return cudaGetLastError();
}

}  // namespace avtp
