// Criterion A (paper §3.3.1): I_v = 1 - cos(h^l_v, h^prior_v) for every visual token,
// plus the fixed-point per-image sums S_i used by the budget rule (§3.3.3).
//
// HBM-bound stream: each visual row of h_cur and h_prior is read once (2 x D x 2
// bytes per token). One warp owns one row at a time and issues 16-byte loads,
// several per lane in flight, accumulating dot, |a|^2 and |b|^2 in fp32.
// h_prior is read with an L2 evict-first policy; h_cur with evict-last, because
// the compaction step reads the kept h_cur rows again right after.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kThreads = 512;
constexpr int kUnroll = 4;  // 16-byte loads per lane per tensor in flight

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint4 ld_stream(const void* ptr, uint64_t pol) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(ptr), "l"(pol));
  return v;
}

__device__ __forceinline__ void accum8(const uint4& a, const uint4& b, float& dot, float& na, float& nb) {
  const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
  const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 fa = __bfloat1622float2(pa[j]);
    const float2 fb = __bfloat1622float2(pb[j]);
    dot = fmaf(fa.x, fb.x, dot);
    dot = fmaf(fa.y, fb.y, dot);
    na = fmaf(fa.x, fa.x, na);
    na = fmaf(fa.y, fa.y, na);
    nb = fmaf(fb.x, fb.x, nb);
    nb = fmaf(fb.y, fb.y, nb);
  }
}

__global__ void __launch_bounds__(kThreads)
k_score_hvar(const __nv_bfloat16* __restrict__ h_cur, int64_t cur_stride, const __nv_bfloat16* __restrict__ h_prior,
             int64_t prior_stride, int D, const int32_t* __restrict__ cu, const int32_t* __restrict__ img_start,
             const int32_t* __restrict__ vis_cu, const int32_t* __restrict__ img_req, int n_img,
             float* __restrict__ scores, int64_t* __restrict__ img_sums, const DevStatus* st) {
  if (!st->layout_ok) return;
  const int lane = threadIdx.x & 31;
  const int warps_per_block = blockDim.x >> 5;
  const int64_t gwarp = static_cast<int64_t>(blockIdx.x) * warps_per_block + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * warps_per_block;
  const int n_vis = vis_cu[n_img];
  const uint64_t pol_first = policy_evict_first();
  const uint64_t pol_last = policy_evict_last();
  int img = 0;  // cached image of the previous row (rows visited in increasing order)
  for (int64_t v = gwarp; v < n_vis; v += nwarps) {
    if (!(vis_cu[img] <= v && v < vis_cu[img + 1])) img = upper_index(vis_cu, n_img, v);
    const int r = img_req[img];
    const int64_t t = static_cast<int64_t>(cu[r]) + img_start[img] + (v - vis_cu[img]);
    const char* pa = reinterpret_cast<const char*>(h_cur + t * cur_stride);
    const char* pb = reinterpret_cast<const char*>(h_prior + t * prior_stride);
    float dot = 0.f, na = 0.f, nb = 0.f;
    const int nvec = D >> 3;  // 16-byte vectors per row
    int c = lane;
    for (; c + 32 * (kUnroll - 1) < nvec; c += 32 * kUnroll) {
      uint4 a[kUnroll], b[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        a[u] = ld_stream(pa + 16 * static_cast<int64_t>(c + 32 * u), pol_last);
        b[u] = ld_stream(pb + 16 * static_cast<int64_t>(c + 32 * u), pol_first);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) accum8(a[u], b[u], dot, na, nb);
    }
    for (; c < nvec; c += 32) {
      const uint4 a = ld_stream(pa + 16 * static_cast<int64_t>(c), pol_last);
      const uint4 b = ld_stream(pb + 16 * static_cast<int64_t>(c), pol_first);
      accum8(a, b, dot, na, nb);
    }
    dot = warp_sum(dot);
    na = warp_sum(na);
    nb = warp_sum(nb);
    if (lane == 0) {
      const float den = fmaxf(sqrtf(na), 1e-8f) * fmaxf(sqrtf(nb), 1e-8f);
      const float I = 1.f - dot / den;
      scores[t] = I;
      atomicAdd(reinterpret_cast<unsigned long long*>(img_sums + img),
                static_cast<unsigned long long>(fixed_point_score(I)));
    }
  }
}

}  // namespace

cudaError_t launch_score_hvar(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                              int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s) {
  if (L.n_images == 0 || L.n_tokens == 0) return cudaSuccess;
  const int warps_per_block = kThreads / 32;
  const int64_t want = (L.n_tokens + warps_per_block - 1) / warps_per_block;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 2;  // 2 x 512 threads per SM
  const int grid = static_cast<int>(want < cap ? want : cap);
  k_score_hvar<<<grid, kThreads, 0, s>>>(
      static_cast<const __nv_bfloat16*>(sa.h_cur), sa.h_cur_stride, static_cast<const __nv_bfloat16*>(sa.h_prior),
      sa.h_prior_stride, sa.hidden, L.cu_seqlens, L.img_start, ws_at<int32_t>(ws, p.vis_cu),
      ws_at<int32_t>(ws, p.img_req), L.n_images, scores, img_sums, ws_at<DevStatus>(ws, p.status));
  return cudaGetLastError();
}

}  // namespace avtp
