// Step 2 as its own kernel (avtp_allocate): one warp per request runs the budget
// rule of avtp_alloc.cuh (paper §3.3.3 adaptive keep ratio, App. A.2 clamps) and
// writes the request's budgets: the register form (a lane per image) for requests of up
// to 32 images, the shared-memory form beyond, as in the fused stage (avtp_prune), which
// runs the same rule inside the selection kernel.
#include "avtp_alloc.cuh"

namespace avtp {
namespace {

constexpr int kMaxWarpsPerCta = 4;
constexpr size_t kSmemBudget = 200 * 1024;

__global__ void __launch_bounds__(kMaxWarpsPerCta * 32, 1)
k_allocate(const int32_t* __restrict__ img_cu, const int32_t* __restrict__ img_len,
           const int64_t* __restrict__ img_sums, const float* __restrict__ keep_ratio, float alpha, float r_min,
           float r_max, int relative, const int32_t* __restrict__ vis_cu, const int32_t* __restrict__ req_budget,
           int32_t* __restrict__ budgets, int R, int m_cap, DevStatus* st) {
  extern __shared__ __align__(16) unsigned char smem[];
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= R || !st->layout_ok) return;
  const int i0 = img_cu[r];
  const int m = img_cu[r + 1] - i0;
  if (m == 0) return;
  const WarpAllocSmem sm = carve_warp_alloc(smem + static_cast<size_t>(warp) * warp_alloc_smem_bytes(m_cap), m_cap);
  if (m <= 32) {
    const bool has = lane < m;
    const int64_t S = has ? img_sums[i0 + lane] : 0;
    const int32_t n = has ? img_len[i0 + lane] : 0;
    const int32_t N = vis_cu[i0 + m] - vis_cu[i0];
    const RatioRule rule = make_ratio_rule(keep_ratio[r], alpha, relative);
    int32_t K = 0;
    const int err = warp_allocate32(sm, m, S, n, recip62(n), req_budget[r], N, recip62(N), rule, alpha, r_min, r_max,
                                    &K);
    if (err != AVTP_OK) {
      if (lane == 0) record_error(st, err, r);
      return;
    }
    if (has) budgets[i0 + lane] = K;
    return;
  }
  for (int j = lane; j < m; j += 32) {
    sm.S[j] = img_sums[i0 + j];
    sm.n[j] = img_len[i0 + j];
  }
  __syncwarp();
  const int32_t N = vis_cu[i0 + m] - vis_cu[i0];
  const int err = warp_allocate(sm, m, req_budget[r], N, keep_ratio[r], alpha, r_min, r_max, relative);
  if (err != AVTP_OK) {
    if (lane == 0) record_error(st, err, r);
    return;
  }
  for (int j = lane; j < m; j += 32) budgets[i0 + j] = sm.K[j];
}

}  // namespace

cudaError_t launch_allocate(const avtp_layout_t& L, const int64_t* img_sums, const avtp_alloc_args_t& aa,
                            int32_t* budgets, void* ws, const WsPlan& p, cudaStream_t s) {
  if (L.n_images == 0) return cudaSuccess;
  const int m_cap = L.n_images < kMaxImagesPerRequest ? L.n_images : kMaxImagesPerRequest;
  const size_t per_warp = warp_alloc_smem_bytes(m_cap);
  int wpc = static_cast<int>(kSmemBudget / per_warp);
  wpc = wpc < 1 ? 1 : (wpc > kMaxWarpsPerCta ? kMaxWarpsPerCta : wpc);
  const size_t smem = wpc * per_warp;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_allocate, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  const int grid = (L.n_requests + wpc - 1) / wpc;
  return launch_kernel(k_allocate, dim3(grid), dim3(32 * wpc), smem, s, /*pdl=*/true, L.img_cu, L.img_len, img_sums,
                       aa.keep_ratio, aa.alpha, aa.r_min, aa.r_max, aa.relative, ws_at<int32_t>(ws, p.vis_cu),
                       ws_at<int32_t>(ws, p.req_budget), budgets, L.n_requests, m_cap,
                       ws_at<DevStatus>(ws, p.status));
}

}  // namespace avtp
