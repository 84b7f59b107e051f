// Step 2: per-image keep budgets (paper §3.3.3 image-aware adaptive ratio; App. A.2 clamps).
//
// One CTA per request. The fp64 part is the ratio formula only, a handful of
// operations per image, each rounded once (explicit _rn intrinsics, so no
// contraction into FMA):
//   Ibar_i   = (S_i * 2^-32) / n_i
//   Ibar_avg = (sum_i S_i * 2^-32) / N_vis                 (token-weighted mean)
//   r_i      = r_base + alpha * (Ibar_i - Ibar_avg)         (relative = 0)
//            = r_base * (1 + alpha * (Ibar_i / Ibar_avg - 1))   (relative = 1)
// Everything after it is exact integer arithmetic on a 2^-40 grid:
//   R_i = rint(clamp(r_i, +-2^20) * 2^40)
//   lambda = min { l : G(l) = sum_i n_i * clamp(R_i + l, R_min, R_max) >= B_r * 2^40 }
//   x_i = n_i * clamp(R_i + lambda), k_i = min(x_i >> 40, n_i), then largest remainder.
// Because G is exact and monotone, lambda is unique whatever the search order;
// here every thread evaluates G at one point and the block narrows the bracket
// by a factor of (threads + 1) per round.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

__device__ __forceinline__ int64_t clamp64(int64_t x, int64_t lo, int64_t hi) {
  return x < lo ? lo : (x > hi ? hi : x);
}

template <typename Op>
__device__ int64_t block_reduce64(int64_t v, int64_t* s_red, Op op) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();  // s_red may still be read by a previous reduction
  if (lane == 0) s_red[warp] = v;
  __syncthreads();
  int64_t r = s_red[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) r = op(r, s_red[w]);
  return r;
}

struct Sum { __device__ int64_t operator()(int64_t a, int64_t b) const { return a + b; } };
struct Min { __device__ int64_t operator()(int64_t a, int64_t b) const { return a < b ? a : b; } };
struct Max { __device__ int64_t operator()(int64_t a, int64_t b) const { return a > b ? a : b; } };

__global__ void __launch_bounds__(kThreads)
k_allocate(const int32_t* __restrict__ img_cu, const int32_t* __restrict__ img_len, const int64_t* __restrict__ img_sums,
           const float* __restrict__ keep_ratio, float alpha, float r_min, float r_max, int relative,
           const int32_t* __restrict__ vis_cu, const int32_t* __restrict__ req_budget, int32_t* __restrict__ budgets,
           int m_cap, DevStatus* st) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int64_t s_red[kWarps];
  __shared__ int64_t s_lo, s_hi;
  if (!st->layout_ok) return;
  const int r = blockIdx.x;
  const int i0 = img_cu[r];
  const int m = img_cu[r + 1] - i0;
  if (m == 0) return;
  int64_t* sR = reinterpret_cast<int64_t*>(smem);  // ratio grid values
  int64_t* sX = sR + m_cap;                        // x_i, then reused for remainders
  int32_t* sN = reinterpret_cast<int32_t*>(sX + m_cap);
  int32_t* sK = sN + m_cap;
  int32_t* sD = sK + m_cap;                        // per-round +-1 decisions

  const int tid = threadIdx.x;
  const int32_t N = vis_cu[i0 + m] - vis_cu[i0];
  const int64_t B = req_budget[r];

  // ---- fp64 ratio formula (one rounding per operation)
  int64_t part = 0;
  for (int j = tid; j < m; j += kThreads) part += img_sums[i0 + j];
  const int64_t total = block_reduce64(part, s_red, Sum());
  const double kScale = 0x1p-32;
  const double ibar_avg = __ddiv_rn(__dmul_rn(__ll2double_rn(total), kScale), static_cast<double>(N));
  const double rb = static_cast<double>(keep_ratio[r]);
  const double al = static_cast<double>(alpha);
  for (int j = tid; j < m; j += kThreads) {
    const int32_t n = img_len[i0 + j];
    const double ibar = __ddiv_rn(__dmul_rn(__ll2double_rn(img_sums[i0 + j]), kScale), static_cast<double>(n));
    double rr;
    if (relative) {
      rr = (ibar_avg == 0.0) ? rb
                             : __dmul_rn(rb, __dadd_rn(1.0, __dmul_rn(al, __dsub_rn(__ddiv_rn(ibar, ibar_avg), 1.0))));
    } else {
      rr = __dadd_rn(rb, __dmul_rn(al, __dsub_rn(ibar, ibar_avg)));
    }
    rr = fmin(fmax(rr, -kRatioLimit), kRatioLimit);
    sR[j] = __double2ll_rn(rr * 0x1p40);  // exact power-of-two scaling
    sN[j] = n;
  }
  __syncthreads();

  // ---- exact water-fill on the 2^-40 grid
  const int64_t Rmin = __double2ll_rn(static_cast<double>(r_min) * 0x1p40);
  const int64_t Rmax = __double2ll_rn(static_cast<double>(r_max) * 0x1p40);
  int64_t mx = INT64_MIN, mn = INT64_MAX;
  for (int j = tid; j < m; j += kThreads) {
    mx = sR[j] > mx ? sR[j] : mx;
    mn = sR[j] < mn ? sR[j] : mn;
  }
  mx = block_reduce64(mx, s_red, Max());
  mn = block_reduce64(mn, s_red, Min());
  const int64_t target = B << kRatioFracBits;
  auto G = [&](int64_t lam) {  // sequential over images; every thread reads the same entry (broadcast)
    int64_t acc = 0;
    for (int j = 0; j < m; ++j) acc += static_cast<int64_t>(sN[j]) * clamp64(sR[j] + lam, Rmin, Rmax);
    return acc;
  };
  int64_t lo = Rmin - mx, hi = Rmax - mn;
  if (tid == 0) {
    if (G(lo) >= target) { s_lo = lo; s_hi = lo; }
    else if (G(hi) < target) { s_lo = hi; s_hi = hi; }
    else { s_lo = lo; s_hi = hi; }
  }
  __syncthreads();
  lo = s_lo;
  hi = s_hi;
  // invariant while hi - lo > 1: G(lo) < target <= G(hi)
  while (hi - lo > 1) {
    const int64_t width = hi - lo;
    const int64_t step = width / (kThreads + 1);
    int64_t p;
    bool active;
    if (step >= 1) { p = lo + step * (tid + 1); active = true; }
    else { p = lo + tid + 1; active = p < hi; }
    int64_t cand_hi = hi, cand_lo = lo;
    if (active) {
      if (G(p) >= target) cand_hi = p; else cand_lo = p;
    }
    const int64_t nhi = block_reduce64(cand_hi, s_red, Min());
    const int64_t nlo = block_reduce64(cand_lo, s_red, Max());
    lo = nlo;
    hi = nhi;
  }
  const int64_t lam = hi;

  // ---- integer budgets and largest remainder
  const int64_t kOneMask = (int64_t(1) << kRatioFracBits) - 1;
  for (int j = tid; j < m; j += kThreads) {
    const int64_t x = static_cast<int64_t>(sN[j]) * clamp64(sR[j] + lam, Rmin, Rmax);
    const int64_t fl = x >> kRatioFracBits;
    sK[j] = static_cast<int32_t>(fl < sN[j] ? fl : sN[j]);
    sX[j] = x & kOneMask;  // remainder
  }
  __syncthreads();
  bool done = false;
  for (int round = 0; round < 64 && !done; ++round) {
    int64_t ks = 0;
    for (int j = tid; j < m; j += kThreads) ks += sK[j];
    const int64_t D = B - block_reduce64(ks, s_red, Sum());
    if (D == 0) { done = true; break; }
    for (int j = tid; j < m; j += kThreads) {
      int dec = 0;
      if (D > 0 && sK[j] < sN[j]) {
        int64_t rank = 0;  // eligible images ahead of j: larger remainder, or equal and lower index
        for (int l = 0; l < m; ++l)
          rank += (sK[l] < sN[l]) && (sX[l] > sX[j] || (sX[l] == sX[j] && l < j));
        dec = rank < D ? 1 : 0;
      } else if (D < 0 && sK[j] > 0) {
        int64_t rank = 0;  // eligible images ahead of j: smaller remainder, or equal and higher index
        for (int l = 0; l < m; ++l)
          rank += (sK[l] > 0) && (sX[l] < sX[j] || (sX[l] == sX[j] && l > j));
        dec = rank < -D ? -1 : 0;
      }
      sD[j] = dec;
    }
    __syncthreads();
    for (int j = tid; j < m; j += kThreads) sK[j] += sD[j];
    __syncthreads();
  }
  if (!done && tid == 0) record_error(st, AVTP_ERR_RANGE, r);
  for (int j = tid; j < m; j += kThreads) budgets[i0 + j] = sK[j];
}

}  // namespace

cudaError_t launch_allocate(const avtp_layout_t& L, const int64_t* img_sums, const avtp_alloc_args_t& aa,
                            int32_t* budgets, void* ws, const WsPlan& p, cudaStream_t s) {
  if (L.n_images == 0) return cudaSuccess;
  const int m_cap = L.n_images < kMaxImagesPerRequest ? L.n_images : kMaxImagesPerRequest;
  const size_t smem = static_cast<size_t>(m_cap) * (8 + 8 + 4 + 4 + 4);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_allocate, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  k_allocate<<<L.n_requests, kThreads, smem, s>>>(L.img_cu, L.img_len, img_sums, aa.keep_ratio, aa.alpha, aa.r_min,
                                                   aa.r_max, aa.relative, ws_at<int32_t>(ws, p.vis_cu),
                                                   ws_at<int32_t>(ws, p.req_budget), budgets, m_cap,
                                                   ws_at<DevStatus>(ws, p.status));
  return cudaGetLastError();
}

}  // namespace avtp
