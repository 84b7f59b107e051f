// Per-request budget rule (paper §3.3.3 adaptive keep ratio, App. A.2 clamps),
// computed by ONE WARP from values staged in that warp's shared memory.
//
// fp64 part (one rounding per operation, explicit _rn intrinsics, no FMA):
//   Ibar_i   = (S_i * 2^-32) / n_i
//   Ibar_avg = (sum_i S_i * 2^-32) / N_vis
//   r_i      = r_base + alpha * (Ibar_i - Ibar_avg)              (relative = 0)
//            = r_base * (1 + alpha * (Ibar_i / Ibar_avg - 1))     (relative = 1; r_base if Ibar_avg == 0)
// exact integer part on the 2^-40 grid:
//   R_i = rint(clamp(r_i, +-2^20) * 2^40), R_min, R_max likewise,
//   G(l) = sum_i n_i * clamp(R_i + l, R_min, R_max),
//   lambda = min { l in [R_min - max R, R_max - min R] : G(l) >= B * 2^40 } (an end of the range if none),
//   x_i = n_i * clamp(R_i + lambda), k_i = min(x_i >> 40, n_i), then largest remainder.
//
// G is continuous, non-decreasing and linear between the breakpoints
// R_min - R_i and R_max - R_i, so for up to kBreakpointImages images lambda is
// found exactly: evaluate G at every breakpoint, take the two that bracket the
// target and solve the linear piece between them with one integer division.
// Beyond that a 32-way multisection gives the same lambda.
//
// Everything is warp-synchronous (shuffles and __syncwarp only): on this part a
// block-wide barrier or a dependent fp64 operation costs far more than the
// arithmetic, so the rule is kept to one warp and a short fp64 chain.
#pragma once

#include "avtp_internal.cuh"

namespace avtp {

constexpr int kBreakpointImages = 64;

__device__ __forceinline__ int64_t clamp64(int64_t x, int64_t lo, int64_t hi) {
  return x < lo ? lo : (x > hi ? hi : x);
}
__device__ __forceinline__ int64_t warp_max64(int64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int64_t u = __shfl_xor_sync(0xffffffffu, v, o);
    v = u > v ? u : v;
  }
  return v;
}
__device__ __forceinline__ int64_t warp_min64(int64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int64_t u = __shfl_xor_sync(0xffffffffu, v, o);
    v = u < v ? u : v;
  }
  return v;
}

// Per-warp scratch, m_cap entries each.
struct WarpAllocSmem {
  int64_t* R;  // ratio grid values
  int64_t* X;  // on entry: S_i (fixed-point sums); on exit: remainders
  int32_t* n;  // on entry: image sizes
  int32_t* K;  // on exit: budgets
};

__host__ __device__ constexpr size_t warp_alloc_smem_bytes(int m_cap) {
  return static_cast<size_t>(m_cap) * (8 + 8 + 4 + 4);
}

__device__ __forceinline__ WarpAllocSmem carve_warp_alloc(unsigned char* base, int m_cap) {
  WarpAllocSmem s;
  s.R = reinterpret_cast<int64_t*>(base);
  s.X = s.R + m_cap;
  s.n = reinterpret_cast<int32_t*>(s.X + m_cap);
  s.K = s.n + m_cap;
  return s;
}

// The grid values of the clamps, rint(r * 2^40) (exact for fp32 inputs >= 2^-17).
__device__ __forceinline__ int64_t ratio_grid(float r) { return __double2ll_rn(static_cast<double>(r) * 0x1p40); }

// All 32 lanes call with identical scalars. sm.X[j] = S_j and sm.n[j] = n_j for j < m on entry.
// Returns false if the rounding loop did not converge (never expected).
static __device__ __noinline__ bool warp_allocate(const WarpAllocSmem& sm, int m, int64_t B, int32_t N, float r_base_f, float alpha_f,
                              int64_t Rmin, int64_t Rmax, int relative) {
  const int lane = threadIdx.x & 31;
  // ---- fp64 ratio formula
  int64_t part = 0;
  for (int j = lane; j < m; j += 32) part += sm.X[j];
  const int64_t total = warp_sum(part);
  const double kScale = 0x1p-32;
  const double ibar_avg = __ddiv_rn(__dmul_rn(__ll2double_rn(total), kScale), static_cast<double>(N));
  const double rb = static_cast<double>(r_base_f);
  const double al = static_cast<double>(alpha_f);
  int64_t mx = INT64_MIN, mn = INT64_MAX;
  for (int j = lane; j < m; j += 32) {
    const double ibar = __ddiv_rn(__dmul_rn(__ll2double_rn(sm.X[j]), kScale), static_cast<double>(sm.n[j]));
    double rr;
    if (relative) {
      rr = (ibar_avg == 0.0) ? rb
                             : __dmul_rn(rb, __dadd_rn(1.0, __dmul_rn(al, __dsub_rn(__ddiv_rn(ibar, ibar_avg), 1.0))));
    } else {
      rr = __dadd_rn(rb, __dmul_rn(al, __dsub_rn(ibar, ibar_avg)));
    }
    rr = fmin(fmax(rr, -kRatioLimit), kRatioLimit);
    const int64_t g = __double2ll_rn(rr * 0x1p40);  // exact power-of-two scaling
    sm.R[j] = g;
    mx = g > mx ? g : mx;
    mn = g < mn ? g : mn;
  }
  mx = warp_max64(mx);
  mn = warp_min64(mn);
  __syncwarp();

  // ---- exact water-fill
  const int64_t target = B << kRatioFracBits;
  auto G = [&](int64_t lam) {
    int64_t acc = 0;
    for (int j = 0; j < m; ++j) acc += static_cast<int64_t>(sm.n[j]) * clamp64(sm.R[j] + lam, Rmin, Rmax);
    return acc;
  };
  const int64_t Llo = Rmin - mx, Lhi = Rmax - mn;
  int64_t lam;
  if (m <= kBreakpointImages) {
    int64_t c_lo = INT64_MIN, c_hi = INT64_MAX, g_lo = 0, g_hi = 0;
    for (int c = lane; c < 2 * m; c += 32) {
      const int j = c >> 1;
      const int64_t cand = (c & 1) ? Rmax - sm.R[j] : Rmin - sm.R[j];
      const int64_t g = G(cand);
      if (g < target) {
        if (cand > c_lo) { c_lo = cand; g_lo = g; }
      } else if (cand < c_hi) {
        c_hi = cand;
        g_hi = g;
      }
    }
    const int64_t best_lo = warp_max64(c_lo);
    const int64_t best_hi = warp_min64(c_hi);
    if (best_hi == INT64_MAX) {
      lam = Lhi;  // G < target everywhere: the upper end
    } else if (best_lo == INT64_MIN) {
      lam = Llo;  // G >= target everywhere: the lower end
    } else {
      // fetch G at the bracketing breakpoints from a lane that holds it
      const int src_lo = __ffs(__ballot_sync(0xffffffffu, c_lo == best_lo)) - 1;
      const int src_hi = __ffs(__ballot_sync(0xffffffffu, c_hi == best_hi)) - 1;
      const int64_t G_lo = __shfl_sync(0xffffffffu, g_lo, src_lo);
      const int64_t G_hi = __shfl_sync(0xffffffffu, g_hi, src_hi);
      // G is linear on [best_lo, best_hi] with integer slope s >= 1
      const int64_t s = (G_hi - G_lo) / (best_hi - best_lo);
      const int64_t need = target - G_lo;  // > 0
      lam = best_lo + (need + s - 1) / s;
    }
  } else {
    // multisection: every lane evaluates one point per round
    int64_t lo = Llo, hi = Lhi;
    if (G(lo) >= target) hi = lo;
    else if (G(hi) < target) lo = hi;
    if (lo == hi) {
      lam = lo;
    } else {
      while (hi - lo > 1) {  // invariant: G(lo) < target <= G(hi)
        const int64_t width = hi - lo;
        const int64_t step = width / 33;
        int64_t p;
        bool active;
        if (step >= 1) { p = lo + step * (lane + 1); active = true; }
        else { p = lo + lane + 1; active = p < hi; }
        int64_t cand_hi = hi, cand_lo = lo;
        if (active) {
          if (G(p) >= target) cand_hi = p; else cand_lo = p;
        }
        hi = warp_min64(cand_hi);
        lo = warp_max64(cand_lo);
      }
      lam = hi;
    }
  }

  // ---- integer budgets and largest remainder
  const int64_t kFracMask = (int64_t(1) << kRatioFracBits) - 1;
  for (int j = lane; j < m; j += 32) {
    const int64_t x = static_cast<int64_t>(sm.n[j]) * clamp64(sm.R[j] + lam, Rmin, Rmax);
    const int64_t fl = x >> kRatioFracBits;
    sm.K[j] = static_cast<int32_t>(fl < sm.n[j] ? fl : sm.n[j]);
    sm.X[j] = x & kFracMask;
  }
  __syncwarp();
  for (int round = 0; round < 64; ++round) {
    int64_t ks = 0;
    for (int j = lane; j < m; j += 32) ks += sm.K[j];
    const int64_t D = B - warp_sum(ks);
    if (D == 0) return true;
    // decide every image from the same snapshot of K (sm.R is free by now), then apply
    for (int j = lane; j < m; j += 32) {
      int dec = 0;
      if (D > 0 && sm.K[j] < sm.n[j]) {
        int64_t rank = 0;  // eligible images ahead of j: larger remainder, or equal and lower index
        for (int l = 0; l < m; ++l)
          rank += (sm.K[l] < sm.n[l]) && (sm.X[l] > sm.X[j] || (sm.X[l] == sm.X[j] && l < j));
        dec = rank < D ? 1 : 0;
      } else if (D < 0 && sm.K[j] > 0) {
        int64_t rank = 0;  // eligible images ahead of j: smaller remainder, or equal and higher index
        for (int l = 0; l < m; ++l)
          rank += (sm.K[l] > 0) && (sm.X[l] < sm.X[j] || (sm.X[l] == sm.X[j] && l > j));
        dec = rank < -D ? -1 : 0;
      }
      sm.R[j] = dec;
    }
    __syncwarp();
    for (int j = lane; j < m; j += 32) sm.K[j] += static_cast<int32_t>(sm.R[j]);
    __syncwarp();
  }
  return false;
}

// lambda from the breakpoints, for warp_allocate32 when a clamp binds near the
// unclamped solution. Out of line: it is the rare case, and its code is only
// fetched when it runs.
static __device__ __noinline__ int64_t breakpoint_lambda32(int m, int64_t R, int64_t nl, bool has, int64_t target,
                                                    int64_t Rmin, int64_t Rmax, int64_t mx, int64_t mn) {
  int64_t lam;
  auto G = [&](int64_t c) {
    int64_t acc = 0;
#pragma unroll 1
    for (int j = 0; j < m; ++j) {
      const int64_t Rj = __shfl_sync(0xffffffffu, R, j);
      const int64_t nj = __shfl_sync(0xffffffffu, nl, j);
      acc += nj * clamp64(Rj + c, Rmin, Rmax);
    }
    return acc;
  };
  // every lane evaluates its two breakpoints (all lanes take part in the shuffles)
  const int64_t cl = Rmin - R, ch = Rmax - R;
  const int64_t gl = G(cl), gh = G(ch);
  int64_t c_lo = INT64_MIN, c_hi = INT64_MAX, g_lo = 0, g_hi = 0;
  if (has) {
    if (gl < target) { c_lo = cl; g_lo = gl; } else { c_hi = cl; g_hi = gl; }
    if (gh < target) {
      if (ch > c_lo) { c_lo = ch; g_lo = gh; }
    } else if (ch < c_hi) {
      c_hi = ch;
      g_hi = gh;
    }
  }
  const int64_t best_lo = warp_max64(c_lo);
  const int64_t best_hi = warp_min64(c_hi);
  if (best_hi == INT64_MAX) {
    lam = Rmax - mn;
  } else if (best_lo == INT64_MIN) {
    lam = Rmin - mx;
  } else {
    const int src_lo = __ffs(__ballot_sync(0xffffffffu, c_lo == best_lo)) - 1;
    const int src_hi = __ffs(__ballot_sync(0xffffffffu, c_hi == best_hi)) - 1;
    const int64_t G_lo = __shfl_sync(0xffffffffu, g_lo, src_lo);
    const int64_t G_hi = __shfl_sync(0xffffffffu, g_hi, src_hi);
    const int64_t sl = (G_hi - G_lo) / (best_hi - best_lo);
    lam = best_lo + (target - G_lo + sl - 1) / sl;
  }
  return lam;
}

// The same rule for requests of at most 32 images, held in registers: lane j owns
// image j (S_j, n_j in; its budget out). Identical results to warp_allocate.
// Fast path for lambda: without clamps G is linear with slope N, so the smallest
// solution is lambda0 = ceil((B * 2^40 - sum n_i R_i) / N); when no clamp binds
// at lambda0 - 1 or lambda0, G is that line on [lambda0 - 1, lambda0] and
// lambda0 is exact. Otherwise the breakpoints decide.
inline __device__ bool warp_allocate32(int m, int64_t S, int32_t n, int64_t B, int32_t N, float r_base_f,
                                       float alpha_f, int64_t Rmin, int64_t Rmax, int relative, int32_t* k_out) {
  const int lane = threadIdx.x & 31;
  const bool has = lane < m;
  // ---- fp64 ratio formula
  const int64_t total = warp_sum(has ? S : int64_t(0));
  const double kScale = 0x1p-32;
  const double ibar_avg = __ddiv_rn(__dmul_rn(__ll2double_rn(total), kScale), static_cast<double>(N));
  const double rb = static_cast<double>(r_base_f);
  const double al = static_cast<double>(alpha_f);
  int64_t R = 0;
  if (has) {
    const double ibar = __ddiv_rn(__dmul_rn(__ll2double_rn(S), kScale), static_cast<double>(n));
    double rr;
    if (relative) {
      rr = (ibar_avg == 0.0) ? rb
                             : __dmul_rn(rb, __dadd_rn(1.0, __dmul_rn(al, __dsub_rn(__ddiv_rn(ibar, ibar_avg), 1.0))));
    } else {
      rr = __dadd_rn(rb, __dmul_rn(al, __dsub_rn(ibar, ibar_avg)));
    }
    rr = fmin(fmax(rr, -kRatioLimit), kRatioLimit);
    R = __double2ll_rn(rr * 0x1p40);
  }
  const int64_t mx = warp_max64(has ? R : INT64_MIN);
  const int64_t mn = warp_min64(has ? R : INT64_MAX);
  const int64_t target = B << kRatioFracBits;
  const int64_t nl = has ? n : 0;

  // ---- exact water-fill
  int64_t lam;
  bool found = false;
  const int64_t kSafe = int64_t(1) << 42;  // keeps n * R and the sums inside int64
  if (mx <= kSafe && mn >= -kSafe) {
    const int64_t snr = warp_sum(nl * R);
    const int64_t num = target - snr;  // smallest lam0 with snr + N * lam0 >= target
    const int64_t lam0 = num >= 0 ? (num + N - 1) / N : -((-num) / N);
    const bool ok = !has || (R + lam0 - 1 >= Rmin && R + lam0 <= Rmax);
    if (__all_sync(0xffffffffu, ok)) {
      lam = lam0;
      found = true;
    }
  }
  if (!found) lam = breakpoint_lambda32(m, R, nl, has, target, Rmin, Rmax, mx, mn);

  // ---- integer budgets and largest remainder
  const int64_t x = nl * clamp64(R + lam, Rmin, Rmax);
  const int64_t fl = x >> kRatioFracBits;
  int32_t K = has ? static_cast<int32_t>(fl < nl ? fl : nl) : 0;
  const int64_t X = x & ((int64_t(1) << kRatioFracBits) - 1);
  for (int round = 0; round < 64; ++round) {
    const int64_t D = B - warp_sum(static_cast<int64_t>(K));
    if (D == 0) {
      *k_out = K;
      return true;
    }
    const bool elig = has && (D > 0 ? K < n : K > 0);
    // remainders are below 2^40: split them so each shuffle moves 32 bits
    const uint32_t xh = static_cast<uint32_t>(X >> 20), xl = static_cast<uint32_t>(X & 0xFFFFF);
    const unsigned elig_mask = __ballot_sync(0xffffffffu, elig);
    int rank = 0;
    // kept rolled: this code runs once per call from a cold instruction cache,
    // where fetching unrolled code costs far more than the loop's latency
#pragma unroll 1
    for (int l = 0; l < m; ++l) {
      const uint32_t h = __shfl_sync(0xffffffffu, xh, l), lo = __shfl_sync(0xffffffffu, xl, l);
      const bool gt = h > xh || (h == xh && lo > xl), eq = h == xh && lo == xl;
      // ahead of this lane: larger remainder (ties: lower index) when adding, the reverse when removing
      const bool ahead = D > 0 ? (gt || (eq && l < lane)) : (!gt && !eq) || (eq && l > lane);
      rank += (((elig_mask >> l) & 1u) && ahead) ? 1 : 0;
    }
    if (elig && rank < (D > 0 ? D : -D)) K += D > 0 ? 1 : -1;
  }
  *k_out = K;
  return false;
}

}  // namespace avtp
