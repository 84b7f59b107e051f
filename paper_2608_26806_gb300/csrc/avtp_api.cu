// C ABI of the AVTP pruning stage: argument validation, workspace plan and the
// launch sequence of every entry point. Kernels live in k_*.cu.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "avtp_fwd.cuh"
#include "avtp_internal.cuh"

namespace avtp {

namespace {

constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

avtp_status_t from_cuda(cudaError_t e) { return e == cudaSuccess ? AVTP_OK : AVTP_ERR_CUDA; }

avtp_status_t check_layout(const avtp_layout_t* L) {
  if (L == nullptr) return AVTP_ERR_INVALID_ARG;
  if (L->n_requests < 1 || L->n_images < 0 || L->n_tokens < 0) return AVTP_ERR_INVALID_ARG;
  if (L->n_tokens > 0x7fffffffLL || L->n_images > 0x7fffffff - L->n_requests) return AVTP_ERR_RANGE;
  if (L->cu_seqlens == nullptr || L->img_cu == nullptr) return AVTP_ERR_INVALID_ARG;
  if (L->n_images > 0 && (L->img_start == nullptr || L->img_len == nullptr)) return AVTP_ERR_INVALID_ARG;
  return AVTP_OK;
}

avtp_status_t check_score_args(const avtp_layout_t* L, const avtp_score_args_t* a) {
  if (a == nullptr) return AVTP_ERR_INVALID_ARG;
  if (a->criterion == AVTP_CRIT_HIDDEN_VARIATION) {
    if (a->h_cur == nullptr || a->h_prior == nullptr) return AVTP_ERR_INVALID_ARG;
    if (a->hidden < 8 || a->hidden % 8 != 0) return AVTP_ERR_UNSUPPORTED;
    if (a->h_cur_stride < a->hidden || a->h_prior_stride < a->hidden) return AVTP_ERR_INVALID_ARG;
    if (a->h_cur_stride % 8 != 0 || a->h_prior_stride % 8 != 0) return AVTP_ERR_UNSUPPORTED;
    if (!aligned16(a->h_cur) || !aligned16(a->h_prior)) return AVTP_ERR_UNSUPPORTED;
    return AVTP_OK;
  }
  if (a->criterion == AVTP_CRIT_TEXT_ATTENTION) {
    if (a->q == nullptr || a->k == nullptr) return AVTP_ERR_INVALID_ARG;
    if (a->head_dim != 64 && a->head_dim != 128) return AVTP_ERR_UNSUPPORTED;
    if (a->n_q_heads < 1 || a->n_kv_heads < 1) return AVTP_ERR_INVALID_ARG;
    if (a->n_q_heads % a->n_kv_heads != 0) return AVTP_ERR_UNSUPPORTED;
    if (a->n_q_heads / a->n_kv_heads > kAttnMaxGroupHeads) return AVTP_ERR_UNSUPPORTED;
    if (a->max_text_tokens < 0) return AVTP_ERR_INVALID_ARG;
    if (attn_plan(*L, *a).rows > 0x7fffffffLL) return AVTP_ERR_RANGE;
    if (a->q_stride < static_cast<int64_t>(a->n_q_heads) * a->head_dim ||
        a->k_stride < static_cast<int64_t>(a->n_kv_heads) * a->head_dim)
      return AVTP_ERR_INVALID_ARG;
    if (a->q_stride % 8 != 0 || a->k_stride % 8 != 0) return AVTP_ERR_UNSUPPORTED;
    if (!aligned16(a->q) || !aligned16(a->k)) return AVTP_ERR_UNSUPPORTED;
    if (!(a->softmax_scale > 0.f) || !isfinite(a->softmax_scale)) return AVTP_ERR_INVALID_ARG;
    if (a->lse != nullptr && a->lse_stride < L->n_tokens) return AVTP_ERR_INVALID_ARG;
    if (a->query_set != AVTP_QUERIES_TEXT && a->query_set != AVTP_QUERIES_LAST) return AVTP_ERR_INVALID_ARG;
    if (a->path != AVTP_PATH_AUTO && a->path != AVTP_PATH_TENSOR && a->path != AVTP_PATH_CUDA)
      return AVTP_ERR_INVALID_ARG;
    if (a->path == AVTP_PATH_TENSOR && a->query_set == AVTP_QUERIES_LAST) return AVTP_ERR_UNSUPPORTED;
    if (attn_uses_cuda_cores(*L, *a) &&
        narrow_plan(*L, *a, attn_plan(*L, *a).max_text).z_elems > kNarrowMaxLogitBytes / 4)
      return AVTP_ERR_RANGE;
    return AVTP_OK;
  }
  return AVTP_ERR_INVALID_ARG;
}

avtp_status_t check_alloc_args(const avtp_alloc_args_t* a) {
  if (a == nullptr || a->keep_ratio == nullptr) return AVTP_ERR_INVALID_ARG;
  if (!(a->alpha >= 0.f && a->alpha <= 1024.f)) return AVTP_ERR_INVALID_ARG;
  if (!(a->r_min >= 0.f && a->r_min <= a->r_max && a->r_max <= 1.f)) return AVTP_ERR_INVALID_ARG;
  if (a->relative != 0 && a->relative != 1) return AVTP_ERR_INVALID_ARG;
  if (!multiple_of_2m32(a->alpha) || !multiple_of_2m32(a->r_min) || !multiple_of_2m32(a->r_max))
    return AVTP_ERR_RANGE;
  return AVTP_OK;
}

// With n_kept = 0 no row is touched, so the pointers of a set may be NULL.
avtp_status_t check_sets(const avtp_rows_t* sets, int32_t n_sets, int64_t n_kept) {
  if (n_sets < 0 || n_sets > AVTP_MAX_ROW_SETS) return AVTP_ERR_INVALID_ARG;
  if (n_sets > 0 && sets == nullptr) return AVTP_ERR_INVALID_ARG;
  for (int i = 0; i < n_sets; ++i) {
    const avtp_rows_t& s = sets[i];
    if (n_kept > 0 && (s.in == nullptr || s.out == nullptr)) return AVTP_ERR_INVALID_ARG;
    if (s.row_bytes < 1 || s.in_stride < s.row_bytes || s.out_stride < s.row_bytes) return AVTP_ERR_INVALID_ARG;
  }
  return AVTP_OK;
}

avtp_status_t check_ws(void* ws, size_t ws_bytes, const WsPlan& p) {
  if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0) return AVTP_ERR_WORKSPACE;
  if (ws_bytes < p.total) return AVTP_ERR_WORKSPACE;
  return AVTP_OK;
}

avtp_status_t record(void* const* events, int i, cudaStream_t s) {
  if (events == nullptr || events[i] == nullptr) return AVTP_OK;
  return from_cuda(cudaEventRecord(static_cast<cudaEvent_t>(events[i]), s));
}

}  // namespace

AttnPlan attn_plan(const avtp_layout_t& L, const avtp_score_args_t& sa) {
  AttnPlan a{};
  const int64_t T = L.n_tokens;
  a.G = sa.n_kv_heads > 0 ? sa.n_q_heads / sa.n_kv_heads : 1;
  a.max_text = (sa.max_text_tokens > 0 && sa.max_text_tokens < T) ? sa.max_text_tokens : T;
  a.rows = a.max_text * a.G;
  // every request's row blocks: ceil(rows_r / 256) <= rows_r / 256 + 1
  a.n_blocks_max = a.rows / kAttnBlockRows + L.n_requests + 1;
  // key tiles: sum_i ceil(n_i / 128) <= N_vis / 128 + n_img
  a.n_ktiles_max = T / kAttnTileM + L.n_images + 1;
  a.Hkv = sa.n_kv_heads;
  a.grid = device_sm_count();
  return a;
}

bool attn_uses_cuda_cores(const avtp_layout_t& L, const avtp_score_args_t& sa) {
  if (sa.path == AVTP_PATH_CUDA || sa.query_set == AVTP_QUERIES_LAST) return true;
  if (sa.path == AVTP_PATH_TENSOR) return false;
  const AttnPlan a = attn_plan(L, sa);
  return a.rows <= kNarrowAutoRows;
}

WsPlan plan_workspace(const avtp_layout_t& L, const avtp_score_args_t* sa) {
  WsPlan p{};
  const size_t R = static_cast<size_t>(L.n_requests), NI = static_cast<size_t>(L.n_images);
  const size_t T = static_cast<size_t>(L.n_tokens);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes);
    return at;
  };
  p.status = take(sizeof(DevStatus));
  p.vis_cu = take((NI + 1) * 4);
  p.img_req = take(NI * 4 + 4);
  p.req_budget = take(R * 4);
  p.img_sums = take(NI * 8 + 8);
  p.scores = take(T * 4 + 4);
  p.scratch = take((NI + 1) * 4);
  if (sa != nullptr && sa->criterion == AVTP_CRIT_TEXT_ATTENTION) {
    const AttnPlan a = attn_plan(L, *sa);
    const size_t Hkv = static_cast<size_t>(sa->n_kv_heads), rows = static_cast<size_t>(a.rows);
    p.text_idx = take(T * 4 + 4);
    p.text_cu = take((R + 1) * 4);
    p.blk_cu = take((R + 1) * 4);
    p.p1s_cu = take((static_cast<size_t>(a.n_blocks_max) + 1) * 4);
    p.p2t_cu = take((static_cast<size_t>(a.n_blocks_max) + 1) * 4);
    p.ktile_cu = take((NI + 1) * 4);
    p.ktile_img = take(static_cast<size_t>(a.n_ktiles_max) * 4);
    p.meta = take(8 * 4);
    if (attn_uses_cuda_cores(L, *sa)) {
      const NarrowPlan np = narrow_plan(L, *sa, a.max_text);
      const size_t nrows = static_cast<size_t>(np.rows);
      p.p1_part = (sa->lse == nullptr) ? take(static_cast<size_t>(np.NS) * nrows * 8 + 8) : 0;
      p.zbuf = take(static_cast<size_t>(np.z_elems) * 4 + 4);
    } else {
      p.qt = take(Hkv * rows * static_cast<size_t>(sa->head_dim) * 2 + 16);
      p.lse_rows = (sa->lse != nullptr) ? take(Hkv * rows * 4 + 4) : 0;
      p.p1_part = (sa->lse == nullptr)
                      ? take(Hkv * static_cast<size_t>(a.n_blocks_max) * kAttnBlockRows * kAttnMaxChunks * 8)
                      : 0;
    }
    p.mass = take(static_cast<size_t>(a.n_ktiles_max) * kAttnTileM * 8);
  }
  p.total = off;
  return p;
}

FwdWs plan_forward_workspace(const avtp_layout_t& L, const avtp_score_args_t& sa, size_t base_bytes) {
  FwdWs f{};
  size_t off = align_up(base_bytes);
  f.Tp = (L.n_tokens + 7) & ~static_cast<int64_t>(7);
  f.vt = off;
  off = align_up(off + static_cast<size_t>(sa.n_kv_heads) * sa.head_dim * static_cast<size_t>(f.Tp) * 2 + 16);
  f.qtile_cu = off;
  off = align_up(off + (static_cast<size_t>(L.n_requests) + 1) * 4);
  f.total = off;
  return f;
}

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = getenv("AVTP_PDL");
    return !(v != nullptr && v[0] == '0');
  }();
  return on;
}

int device_sm_count() {
  static PerDevice sms;
  int n = 0;
  const cudaError_t e = once_per_device(sms, [](int dev, int* v) {
    return cudaDeviceGetAttribute(v, cudaDevAttrMultiProcessorCount, dev);
  }, &n);
  return (e == cudaSuccess && n > 0) ? n : 148;
}

// SMs the scoring kernel leaves to the selection kernel, at most.
constexpr int kMaxReserveSms = 32;

int prune_reserve_sms(const avtp_layout_t& L) {
  if (L.n_tokens > 32768 || L.n_images < 1) return 0;
  const int64_t ctas = prune_warm_ctas(L);
  // one SM per selection CTA (its registers fill most of an SM; two on one SM slowed each
  // other's budget rule) and one for the validation kernel, which runs when the scoring
  // kernel starts: at most kMaxReserveSms, the CTAs beyond start when the scoring
  // kernel's CTAs end
  return static_cast<int>(ctas + 1 < kMaxReserveSms ? ctas + 1 : kMaxReserveSms);
}

int prune_warm_ctas(const avtp_layout_t& L) {
  if (L.n_tokens > 32768 || L.n_images < 1) return 0;
  const int64_t ctas = static_cast<int64_t>(L.n_images) + L.n_requests;
  return ctas <= kMaxWarmCtas ? static_cast<int>(ctas) : 0;
}

}  // namespace avtp

using namespace avtp;

extern "C" {

avtp_status_t avtp_workspace_size(const avtp_layout_t* layout, const avtp_score_args_t* score_args, size_t* bytes) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if (bytes == nullptr) return AVTP_ERR_INVALID_ARG;
  if (score_args != nullptr && (st = check_score_args(layout, score_args)) != AVTP_OK) return st;
  *bytes = plan_workspace(*layout, score_args).total;
  return AVTP_OK;
}


static avtp_status_t score_impl(const avtp_layout_t* L, const avtp_score_args_t* a, float* scores,
                                int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s, int reserve_sms = 0) {
  if (a->criterion == AVTP_CRIT_HIDDEN_VARIATION)
    return from_cuda(launch_score_hvar(*L, *a, scores, img_sums, ws, p, s, reserve_sms));
  if (attn_uses_cuda_cores(*L, *a))
    return from_cuda(launch_score_narrow(*L, *a, scores, img_sums, ws, p, attn_plan(*L, *a), s));
  return from_cuda(launch_score_attn(*L, *a, scores, img_sums, ws, p, s));
}

avtp_status_t avtp_score(const avtp_layout_t* layout, const avtp_score_args_t* args, float* scores,
                         int64_t* img_sums, void* workspace, size_t workspace_bytes, avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if ((st = check_score_args(layout, args)) != AVTP_OK) return st;
  if (scores == nullptr || img_sums == nullptr) return AVTP_ERR_INVALID_ARG;
  const WsPlan p = plan_workspace(*layout, args);
  if ((st = check_ws(workspace, workspace_bytes, p)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = *layout;
  pa.zero_img_sums = img_sums;
  pa.build_text_tiles = args->criterion == AVTP_CRIT_TEXT_ATTENTION;
  if (pa.build_text_tiles) {
    pa.attn = attn_plan(*layout, *args);
  }
  if ((st = from_cuda(launch_prep(pa, workspace, p, s))) != AVTP_OK) return st;
  return score_impl(layout, args, scores, img_sums, workspace, p, s);
}

// The forward's arguments, and the score arguments of its criterion-B side output (the
// caller's, with the LSE the forward writes supplied).
static avtp_status_t forward_args(const avtp_layout_t* L, const avtp_score_args_t* a, const avtp_forward_args_t* f,
                                  avtp_score_args_t* sa_out) {
  if (a == nullptr || f == nullptr) return AVTP_ERR_INVALID_ARG;
  if (a->criterion != AVTP_CRIT_TEXT_ATTENTION || a->lse != nullptr) return AVTP_ERR_INVALID_ARG;
  if (f->v == nullptr || f->o == nullptr || f->lse == nullptr) return AVTP_ERR_INVALID_ARG;
  avtp_score_args_t sa = *a;
  sa.lse = f->lse;
  sa.lse_stride = f->lse_stride;
  avtp_status_t st = check_score_args(L, &sa);
  if (st != AVTP_OK) return st;
  const int64_t Hq = sa.n_q_heads, Hkv = sa.n_kv_heads, d = sa.head_dim;
  if (f->v_stride < Hkv * d || f->o_stride < Hq * d) return AVTP_ERR_INVALID_ARG;
  if (f->v_stride % 8 != 0 || f->o_stride % 4 != 0) return AVTP_ERR_UNSUPPORTED;
  if (!aligned16(f->v) || !aligned16(f->o)) return AVTP_ERR_UNSUPPORTED;
  // query tiles x heads, the forward's grid: (T / 128 + R) * Hq CTAs
  if ((L->n_tokens / 128 + L->n_requests) * Hq > 0x7fffffffLL) return AVTP_ERR_RANGE;
  *sa_out = sa;
  return AVTP_OK;
}

avtp_status_t avtp_forward_workspace_size(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                                          const avtp_forward_args_t* fwd_args, size_t* bytes) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if (bytes == nullptr) return AVTP_ERR_INVALID_ARG;
  avtp_score_args_t sa{};
  if ((st = forward_args(layout, score_args, fwd_args, &sa)) != AVTP_OK) return st;
  *bytes = plan_forward_workspace(*layout, sa, plan_workspace(*layout, &sa).total).total;
  return AVTP_OK;
}

avtp_status_t avtp_attn_forward(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                                const avtp_forward_args_t* fwd_args, float* scores, int64_t* img_sums,
                                void* workspace, size_t workspace_bytes, avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  avtp_score_args_t sa{};
  if ((st = forward_args(layout, score_args, fwd_args, &sa)) != AVTP_OK) return st;
  if ((scores == nullptr) != (img_sums == nullptr)) return AVTP_ERR_INVALID_ARG;
  const WsPlan p = plan_workspace(*layout, &sa);
  const FwdWs f = plan_forward_workspace(*layout, sa, p.total);
  WsPlan whole = p;
  whole.total = f.total;
  if ((st = check_ws(workspace, workspace_bytes, whole)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = *layout;
  pa.zero_img_sums = img_sums;
  pa.build_text_tiles = scores != nullptr;
  if (pa.build_text_tiles) pa.attn = attn_plan(*layout, sa);
  if ((st = from_cuda(launch_prep(pa, workspace, p, s))) != AVTP_OK) return st;
  if ((st = from_cuda(launch_attn_forward(*layout, sa, *fwd_args, workspace, p, f, s))) != AVTP_OK) return st;
  if (scores == nullptr) return AVTP_OK;
  return score_impl(layout, &sa, scores, img_sums, workspace, p, s);
}

avtp_status_t avtp_allocate(const avtp_layout_t* layout, const int64_t* img_sums, const avtp_alloc_args_t* args,
                            int32_t* budgets, int32_t* out_cu_seqlens, void* workspace, size_t workspace_bytes,
                            avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if ((st = check_alloc_args(args)) != AVTP_OK) return st;
  if ((layout->n_images > 0 && (img_sums == nullptr || budgets == nullptr)) || out_cu_seqlens == nullptr)
    return AVTP_ERR_INVALID_ARG;
  const WsPlan p = plan_workspace(*layout, nullptr);
  if ((st = check_ws(workspace, workspace_bytes, p)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = *layout;
  pa.keep_ratio = args->keep_ratio;
  pa.r_min = args->r_min;
  pa.r_max = args->r_max;
  pa.out_cu_seqlens = out_cu_seqlens;
  if ((st = from_cuda(launch_prep(pa, workspace, p, s))) != AVTP_OK) return st;
  return from_cuda(launch_allocate(*layout, img_sums, *args, budgets, workspace, p, s));
}

avtp_status_t avtp_select(const avtp_layout_t* layout, const float* scores, const int32_t* budgets,
                          const int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, void* workspace,
                          size_t workspace_bytes, avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if (out_cu_seqlens == nullptr || n_kept < 0 || (n_kept > 0 && kept_idx == nullptr)) return AVTP_ERR_INVALID_ARG;
  if (layout->n_images > 0 && (scores == nullptr || budgets == nullptr)) return AVTP_ERR_INVALID_ARG;
  const WsPlan p = plan_workspace(*layout, nullptr);
  if ((st = check_ws(workspace, workspace_bytes, p)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = *layout;
  if ((st = from_cuda(launch_prep(pa, workspace, p, s))) != AVTP_OK) return st;
  return from_cuda(launch_select(*layout, scores, budgets, out_cu_seqlens, kept_idx, n_kept, workspace, p, s));
}

avtp_status_t avtp_compact(const int32_t* kept_idx, int64_t n_kept, int64_t n_tokens, const avtp_rows_t* sets,
                           int32_t n_sets, void* workspace, size_t workspace_bytes, avtp_stream_t stream) {
  avtp_status_t st = check_sets(sets, n_sets, n_kept);
  if (st != AVTP_OK) return st;
  if (n_kept < 0 || n_tokens < 0 || (n_kept > 0 && kept_idx == nullptr)) return AVTP_ERR_INVALID_ARG;
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1)) != 0 ||
      workspace_bytes < sizeof(DevStatus))
    return AVTP_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  WsPlan p{};
  p.status = 0;
  if ((st = from_cuda(cudaMemsetAsync(workspace, 0, sizeof(DevStatus), s))) != AVTP_OK) return st;
  return from_cuda(launch_compact(kept_idx, n_kept, n_tokens, sets, n_sets, workspace, p, s));
}

avtp_status_t avtp_prune(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                         const avtp_alloc_args_t* alloc_args, float* scores, int64_t* img_sums, int32_t* budgets,
                         int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, const avtp_rows_t* sets,
                         int32_t n_sets, void* workspace, size_t workspace_bytes, void* const* step_events,
                         avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if ((st = check_score_args(layout, score_args)) != AVTP_OK) return st;
  if ((st = check_alloc_args(alloc_args)) != AVTP_OK) return st;
  if ((st = check_sets(sets, n_sets, n_kept)) != AVTP_OK) return st;
  if (out_cu_seqlens == nullptr || n_kept < 0 || (n_kept > 0 && kept_idx == nullptr)) return AVTP_ERR_INVALID_ARG;
  if (layout->n_images > 0 && budgets == nullptr) return AVTP_ERR_INVALID_ARG;
  const WsPlan p = plan_workspace(*layout, score_args);
  if ((st = check_ws(workspace, workspace_bytes, p)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  float* sc = scores != nullptr ? scores : ws_at<float>(workspace, p.scores);
  int64_t* sums = img_sums != nullptr ? img_sums : ws_at<int64_t>(workspace, p.img_sums);

  if ((st = record(step_events, 0, s)) != AVTP_OK) return st;
#ifdef AVTP_TIMELINE
  // the timeline words: earliest stamps start at all ones, latest at zero
  char* tl = static_cast<char*>(workspace) + p.status + kTimelineOffset;
  if (cudaMemsetAsync(tl, 0xff, kTlEvents * sizeof(uint64_t), s) != cudaSuccess ||
      cudaMemsetAsync(tl + kTlEvents * sizeof(uint64_t), 0, kTlEvents * sizeof(uint64_t), s) != cudaSuccess)
    return AVTP_ERR_CUDA;
#endif
  PrepArgs pa{};
  pa.L = *layout;
  pa.keep_ratio = alloc_args->keep_ratio;
  pa.r_min = alloc_args->r_min;
  pa.r_max = alloc_args->r_max;
  pa.out_cu_seqlens = out_cu_seqlens;
  pa.zero_img_sums = sums;
  pa.build_text_tiles = score_args->criterion == AVTP_CRIT_TEXT_ATTENTION;
  if (pa.build_text_tiles) {
    pa.attn = attn_plan(*layout, *score_args);
  }
  if ((st = from_cuda(launch_prep(pa, workspace, p, s))) != AVTP_OK) return st;
  if ((st = record(step_events, 1, s)) != AVTP_OK) return st;
  const int reserve = score_args->criterion == AVTP_CRIT_HIDDEN_VARIATION ? prune_reserve_sms(*layout) : 0;
  if ((st = score_impl(layout, score_args, sc, sums, workspace, p, s, reserve)) != AVTP_OK) return st;
  if ((st = record(step_events, 2, s)) != AVTP_OK) return st;
  const int warm = score_args->criterion == AVTP_CRIT_HIDDEN_VARIATION ? prune_warm_ctas(*layout) : 0;
  if ((st = from_cuda(launch_alloc_select(*layout, sums, *alloc_args, budgets, sc, out_cu_seqlens, kept_idx, n_kept,
                                          workspace, p, s, warm))) != AVTP_OK)
    return st;
  if ((st = record(step_events, 3, s)) != AVTP_OK) return st;
  if ((st = from_cuda(launch_compact(kept_idx, n_kept, layout->n_tokens, sets, n_sets, workspace, p, s))) != AVTP_OK)
    return st;
  return record(step_events, 4, s);
}

int64_t avtp_kept_count_host(const int32_t* cu_seqlens, const int32_t* img_cu, const int32_t* img_len,
                             const float* keep_ratio, int32_t n_requests) {
  if (cu_seqlens == nullptr || img_cu == nullptr || keep_ratio == nullptr || n_requests < 1) return -1;
  if (img_cu[n_requests] > 0 && img_len == nullptr) return -1;
  int64_t total = 0;
  for (int r = 0; r < n_requests; ++r) {
    int64_t nvis = 0;
    if (img_cu[r + 1] < img_cu[r] || cu_seqlens[r + 1] < cu_seqlens[r]) return -1;
    for (int i = img_cu[r]; i < img_cu[r + 1]; ++i) nvis += img_len[i];
    const float kr = keep_ratio[r];
    if (!(kr >= 0.f && kr <= 1.f)) return -1;
    // floor(kr * N + 0.5) with each operation rounded once (built with FMA contraction off)
    volatile double prod = static_cast<double>(kr) * static_cast<double>(nvis);
    const double x = prod + 0.5;
    total += static_cast<int64_t>(floor(x)) + (static_cast<int64_t>(cu_seqlens[r + 1]) - cu_seqlens[r] - nvis);
  }
  return total;
}

avtp_status_t avtp_pruned_layout(const avtp_layout_t* layout, const int32_t* budgets, int32_t* out_img_start,
                                 int32_t* out_img_len, void* workspace, size_t workspace_bytes, avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if (layout->n_images > 0 && (budgets == nullptr || out_img_start == nullptr || out_img_len == nullptr))
    return AVTP_ERR_INVALID_ARG;
  const WsPlan p = plan_workspace(*layout, nullptr);
  if ((st = check_ws(workspace, workspace_bytes, p)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = *layout;
  pa.pl_budgets = budgets;
  pa.pl_out_start = out_img_start;
  pa.pl_out_len = out_img_len;
  return from_cuda(launch_prep(pa, workspace, p, s));
}

int64_t avtp_kept_count_vis_host(const int32_t* cu_seqlens, const int32_t* n_vis, const float* keep_ratio,
                                 int32_t n_requests, int32_t* out_cu_seqlens, int32_t* out_n_vis) {
  if (cu_seqlens == nullptr || n_vis == nullptr || keep_ratio == nullptr || n_requests < 1) return -1;
  int64_t total = 0;
  if (out_cu_seqlens != nullptr) out_cu_seqlens[0] = 0;
  for (int r = 0; r < n_requests; ++r) {
    const int64_t Tr = static_cast<int64_t>(cu_seqlens[r + 1]) - cu_seqlens[r];
    if (Tr < 0 || n_vis[r] < 0 || n_vis[r] > Tr) return -1;
    const float kr = keep_ratio[r];
    if (!(kr >= 0.f && kr <= 1.f)) return -1;
    // floor(kr * N + 0.5) with each operation rounded once (built with FMA contraction off)
    volatile double prod = static_cast<double>(kr) * static_cast<double>(n_vis[r]);
    const double x = prod + 0.5;
    const int64_t kept_vis = static_cast<int64_t>(floor(x));
    total += kept_vis + (Tr - n_vis[r]);
    if (total > 0x7fffffffLL) return -1;
    if (out_cu_seqlens != nullptr) out_cu_seqlens[r + 1] = static_cast<int32_t>(total);
    if (out_n_vis != nullptr) out_n_vis[r] = static_cast<int32_t>(kept_vis);
  }
  return total;
}

avtp_status_t avtp_wait_selftest(int64_t limit_ns, int32_t arrive, void* workspace, size_t workspace_bytes,
                                 avtp_stream_t stream) {
  if (limit_ns < 1000 || limit_ns > 10000000000LL) return AVTP_ERR_INVALID_ARG;
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1)) != 0 ||
      workspace_bytes < sizeof(DevStatus))
    return AVTP_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  avtp_status_t st = from_cuda(cudaMemsetAsync(workspace, 0, sizeof(DevStatus), s));
  if (st != AVTP_OK) return st;
  return from_cuda(launch_wait_selftest(static_cast<uint64_t>(limit_ns), arrive != 0, workspace, s));
}

avtp_status_t avtp_layer_attention(const avtp_layout_t* layout, const int64_t* img_sums, int64_t* A,
                                   int32_t n_layers, int32_t layer, void* workspace, size_t workspace_bytes,
                                   avtp_stream_t stream) {
  avtp_status_t st = check_layout(layout);
  if (st != AVTP_OK) return st;
  if (A == nullptr || (layout->n_images > 0 && img_sums == nullptr)) return AVTP_ERR_INVALID_ARG;
  if (n_layers < 1 || layer < 0 || layer >= n_layers) return AVTP_ERR_INVALID_ARG;
  if (n_layers > AVTP_MAX_LAYERS) return AVTP_ERR_RANGE;
  const WsPlan p = plan_workspace(*layout, nullptr);
  if ((st = check_ws(workspace, workspace_bytes, p)) != AVTP_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = *layout;
  if ((st = from_cuda(launch_prep(pa, workspace, p, s))) != AVTP_OK) return st;
  return from_cuda(launch_layer_attention(*layout, img_sums, A, n_layers, layer, workspace, p, s));
}

avtp_status_t avtp_layer_select(const int64_t* A, int32_t n_samples, int32_t n_layers, int32_t k, int64_t* rank_sum,
                                int32_t* top_layers, avtp_stream_t stream) {
  if (A == nullptr || rank_sum == nullptr || top_layers == nullptr) return AVTP_ERR_INVALID_ARG;
  if (n_samples < 1 || n_layers < 1 || k < 1 || k > n_layers) return AVTP_ERR_INVALID_ARG;
  if (n_layers > AVTP_MAX_LAYERS) return AVTP_ERR_RANGE;
  return from_cuda(launch_layer_select(A, n_samples, n_layers, k, rank_sum, top_layers,
                                       reinterpret_cast<cudaStream_t>(stream)));
}

avtp_status_t avtp_read_device_status(const void* workspace, avtp_stream_t stream, int32_t* out) {
  if (workspace == nullptr || out == nullptr) return AVTP_ERR_INVALID_ARG;
  DevStatus h{};
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(&h, workspace, sizeof(h), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return AVTP_ERR_CUDA;
  *out = h.code;
  return AVTP_OK;
}

const char* avtp_status_string(int32_t status) {
  switch (status) {
    case AVTP_OK: return "ok";
    case AVTP_ERR_INVALID_ARG: return "invalid argument";
    case AVTP_ERR_UNSUPPORTED: return "unsupported configuration";
    case AVTP_ERR_RANGE: return "size outside the supported range";
    case AVTP_ERR_CUDA: return "CUDA runtime error";
    case AVTP_ERR_TIMEOUT: return "device wait timed out";
    case AVTP_ERR_DEVICE_INPUT: return "device data failed validation";
    case AVTP_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    default: return "unknown status";
  }
}

int32_t avtp_version(void) { return 100; }

}  // extern "C"
