// Per-request budget rule (paper §3.3.3 adaptive keep ratio, App. A.2 clamps),
// computed by ONE WARP, in exact integer arithmetic on a 2^-40 ratio grid.
//
// Ratios (S_i in units of 2^-32, each product exact, rounded once to nearest, ties up):
//   Ibar_i   = round(S_i * floor(2^62 / n_i) / 2^62)
//   Ibar_avg = round(sum_i S_i * floor(2^62 / N_vis) / 2^62)
//   R_i = R_base + round(alpha * (Ibar_i - Ibar_avg) * 2^8)                       (relative = 0)
//   R_i = R_base + round(r_base * alpha * q_i),                                    (relative = 1)
//         q_i = sgn(Ibar_avg) * round((Ibar_i - Ibar_avg) * floor(2^62 / |Ibar_avg|) / 2^22),
//         saturated to +-2^60 (R_i = R_base when Ibar_avg == 0)
//   with R_base = rint(r_base * 2^40), fp32 alpha and r_base taken as exact M * 2^E,
//   and R_i saturated to +-2^60. R_min, R_max = rint(r_min * 2^40), rint(r_max * 2^40).
// Water-fill and rounding:
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
// block-wide barrier or a dependent fp64 operation or division costs far more
// than the arithmetic, so the reciprocals are taken before the sums are known
// and the rest is integer multiplies and shifts.
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

constexpr int kRecipBits = 62;
constexpr int64_t kGridSat = int64_t(1) << 60;   // ratios saturate here on the grid
constexpr int kSumMagnitudeBits = 42;            // |S_i| <= n_i * 2^42 (scores clamped to +-2^10)

// floor(2^62 / n) for n >= 1 (0 for n <= 0, which only unused lanes pass).
__device__ __forceinline__ int64_t recip62(int64_t n) {
  return n > 0 ? static_cast<int64_t>((uint64_t(1) << kRecipBits) / static_cast<uint64_t>(n)) : 0;
}

// floor(x / 2^s + 1/2) for 1 <= s, saturated to +-lim.
__device__ __forceinline__ int64_t round_shift_sat(__int128 x, int s, int64_t lim) {
  if (s > 120) return 0;  // every x passed here is below 2^110 in magnitude
  const __int128 y = (x + (static_cast<__int128>(1) << (s - 1))) >> s;
  return y > lim ? lim : (y < -lim ? -lim : static_cast<int64_t>(y));
}

// The fp32 value v as M * 2^E exactly, |M| < 2^24.
__device__ __forceinline__ void fp32_parts(float v, int64_t* M, int* E) {
  const uint32_t b = __float_as_uint(v);
  const int e8 = (b >> 23) & 0xff;
  const int64_t mag = (b & 0x7fffff) | (e8 ? 0x800000 : 0);
  *M = (b >> 31) ? -mag : mag;
  *E = e8 ? e8 - 150 : -149;
}

// The parts of the ratio rule that do not depend on the sums. alpha in [0, 1024]
// and r_base in [0, 1] (validated before any launch) keep `shift` >= 5.
struct RatioRule {
  int64_t Rb;    // rint(r_base * 2^40)
  int64_t coef;  // alpha (additive) or r_base * alpha (relative) is coef * 2^-shift on the grid
  int shift;
  int relative;
};

__device__ __forceinline__ RatioRule make_ratio_rule(float r_base, float alpha, int relative) {
  RatioRule q;
  q.Rb = ratio_grid(r_base);
  int64_t A, Bm;
  int E, Be;
  fp32_parts(alpha, &A, &E);
  fp32_parts(r_base, &Bm, &Be);
  q.relative = relative;
  if (relative) {
    q.coef = A * Bm;
    q.shift = -(E + Be);
  } else {
    q.coef = A;
    q.shift = -(E + kRatioFracBits - kFxFracBits);
  }
  return q;
}

// Ibar on the 2^-32 grid: round(S * floor(2^62 / n) / 2^62), exact for |S| <= n * 2^42.
__device__ __forceinline__ int64_t grid_mean(int64_t S, int64_t inv_n) {
  return round_shift_sat(static_cast<__int128>(S) * inv_n, kRecipBits, INT64_MAX);
}

// ceil(a / N) for N >= 1 and |a| < 2^62, from inv_N = floor(2^62 / N): the product gives
// the quotient to within one, which a multiply-back corrects (no division instruction).
__device__ __forceinline__ int64_t ceil_div_recip(int64_t a, int64_t N, int64_t inv_N) {
  const uint64_t u = static_cast<uint64_t>(a >= 0 ? a : -a);
  uint64_t q = static_cast<uint64_t>((static_cast<unsigned __int128>(u) * static_cast<uint64_t>(inv_N)) >> kRecipBits);
  uint64_t r = u - q * static_cast<uint64_t>(N);  // q <= floor(u / N) <= q + 2
  if (r >= static_cast<uint64_t>(N)) { ++q; r -= static_cast<uint64_t>(N); }
  if (r >= static_cast<uint64_t>(N)) { ++q; r -= static_cast<uint64_t>(N); }
  // now q = floor(u / N), r = u mod N
  return a >= 0 ? static_cast<int64_t>(q + (r != 0 ? 1 : 0)) : -static_cast<int64_t>(q);
}

// R_i from Ibar_i, Ibar_avg and (relative rule only) floor(2^62 / |Ibar_avg|).
__device__ __forceinline__ int64_t grid_ratio(const RatioRule& q, int64_t ibar, int64_t avg, int64_t inv_avg) {
  const int64_t d = ibar - avg;
  int64_t delta;
  if (!q.relative) {
    delta = round_shift_sat(static_cast<__int128>(q.coef) * d, q.shift, kGridSat * 2);
  } else if (avg == 0) {
    delta = 0;
  } else {
    int64_t t = round_shift_sat(static_cast<__int128>(d) * inv_avg, kRecipBits - kRatioFracBits, kGridSat);
    t = avg > 0 ? t : -t;
    delta = round_shift_sat(static_cast<__int128>(q.coef) * t, q.shift, kGridSat * 2);
  }
  return clamp64(q.Rb + delta, -kGridSat, kGridSat);
}

// All 32 lanes call with identical scalars. sm.X[j] = S_j and sm.n[j] = n_j for j < m on entry.
// Returns AVTP_OK, AVTP_ERR_DEVICE_INPUT for a sum beyond n_j * 2^42, or AVTP_ERR_RANGE
// if the rounding loop did not converge (never expected).
static __device__ __noinline__ int warp_allocate(const WarpAllocSmem& sm, int m, int64_t B, int32_t N, float r_base_f, float alpha_f,
                              int64_t Rmin, int64_t Rmax, int relative) {
  const int lane = threadIdx.x & 31;
  // ---- ratios on the grid
  int64_t part = 0;
  bool bad = false;
  for (int j = lane; j < m; j += 32) {
    const int64_t S = sm.X[j], lim = static_cast<int64_t>(sm.n[j]) << kSumMagnitudeBits;
    bad |= S > lim || S < -lim;
    part += S;
  }
  if (__any_sync(0xffffffffu, bad)) return AVTP_ERR_DEVICE_INPUT;
  const int64_t avg = grid_mean(warp_sum(part), recip62(N));
  const int64_t inv_avg = (relative && avg != 0) ? recip62(avg > 0 ? avg : -avg) : 0;
  const RatioRule rule = make_ratio_rule(r_base_f, alpha_f, relative);
  int64_t mx = INT64_MIN, mn = INT64_MAX;
  for (int j = lane; j < m; j += 32) {
    const int64_t g = grid_ratio(rule, grid_mean(sm.X[j], recip62(sm.n[j])), avg, inv_avg);
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
    if (D == 0) return AVTP_OK;
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
  return AVTP_ERR_RANGE;
}

// The k-th largest (1 <= k <= 32) of the 32 lanes' values: a bitonic sort across the
// warp (15 compare-exchange stages by shuffle), then one broadcast. Out of line and
// rolled: it is fetched once per call from a cold instruction cache.
static __device__ __noinline__ uint64_t warp_kth_largest(uint64_t v, int k) {
  const int lane = threadIdx.x & 31;
#pragma unroll 1
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll 1
    for (int j = size >> 1; j > 0; j >>= 1) {
      const uint64_t p = __shfl_xor_sync(0xffffffffu, v, j);
      // descending overall: the lower lane of a pair keeps the larger value in blocks
      // whose `size` bit is clear, the smaller one otherwise
      const bool keep_max = ((lane & j) == 0) == ((lane & size) == 0);
      v = keep_max ? (p > v ? p : v) : (p < v ? p : v);
    }
  }
  return __shfl_sync(0xffffffffu, v, k - 1);
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
// image j (S_j, n_j in; its budget out). Identical results and status to warp_allocate.
// Out of line so that a warm-up call and the real one share the same code.
// inv_n = floor(2^62 / n_j) and inv_N = floor(2^62 / N) come from the caller, which
// can take them before the sums are ready; after that no division is left on the
// common path.
// Fast path for lambda: without clamps G is linear with slope N, so the smallest
// solution is lambda0 = ceil((B * 2^40 - sum n_i R_i) / N); when no clamp binds
// at lambda0 - 1 or lambda0, G is that line on [lambda0 - 1, lambda0] and
// lambda0 is exact. Otherwise the breakpoints decide.
static __device__ __noinline__ int warp_allocate32(int m, int64_t S, int32_t n, int64_t inv_n, int64_t B, int32_t N,
                                                   int64_t inv_N, const RatioRule& rule, int64_t Rmin, int64_t Rmax,
                                                   int32_t* k_out) {
  const int lane = threadIdx.x & 31;
  const bool has = lane < m;
  // ---- ratios on the grid
  const int64_t lim = static_cast<int64_t>(n) << kSumMagnitudeBits;
  if (__any_sync(0xffffffffu, has && (S > lim || S < -lim))) return AVTP_ERR_DEVICE_INPUT;
  const int64_t avg = grid_mean(warp_sum(has ? S : int64_t(0)), inv_N);
  const int64_t inv_avg = (rule.relative && avg != 0) ? recip62(avg > 0 ? avg : -avg) : 0;
  const int64_t R = has ? grid_ratio(rule, grid_mean(S, inv_n), avg, inv_avg) : 0;
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
    const int64_t num = target - snr;  // smallest lam0 with snr + N * lam0 >= target: ceil(num / N)
    const int64_t lam0 = ceil_div_recip(num, N, inv_N);
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
      return AVTP_OK;
    }
    const bool elig = has && (D > 0 ? K < n : K > 0);
    // One unique key per eligible lane, larger = served first: adding, larger
    // remainder then lower index; removing, smaller remainder then higher index.
    // Remainders are below 2^40, so a key fits in 45 bits; ineligible lanes get 0.
    const uint64_t rem = static_cast<uint64_t>(X);
    const uint64_t key = !elig ? 0ull
                         : (D > 0 ? (rem << 5) | static_cast<uint64_t>(31 - lane)
                                  : (((uint64_t(1) << kRatioFracBits) - 1 - rem) << 5) | static_cast<uint64_t>(lane));
    // the |D|-th largest key (0 when fewer lanes are eligible): every eligible lane at
    // or above it moves by one
    const uint64_t thr = warp_kth_largest(key, static_cast<int>(D > 0 ? (D < 32 ? D : 32) : (-D < 32 ? -D : 32)));
    if (elig && key >= thr) K += D > 0 ? 1 : -1;
  }
  *k_out = K;
  return AVTP_ERR_RANGE;
}

}  // namespace avtp
