// Per-request budget rule (paper §3.3.3 adaptive keep ratio, App. A.2 clamps), run by
// ONE WARP. Two stages:
//  1. An integer approximation on a 2^-40 ratio grid proposes the water-fill shift:
//       Ibar_i   ~ round(S_i * floor(2^62 / n_i) / 2^62)            (units of 2^-32)
//       Ibar_avg ~ round(sum_i S_i * floor(2^62 / N_vis) / 2^62)
//       R_i = R_base + round(alpha * (Ibar_i - Ibar_avg) * 2^8)                 (additive)
//       R_i = R_base + round(r_base * alpha * q_i),                              (relative)
//         q_i = sgn(Ibar_avg) * round((Ibar_i - Ibar_avg) * floor(2^62 / |Ibar_avg|) / 2^22)
//       lambda = min { l : sum_i n_i * clamp(R_i + l, R_min, R_max) >= B * 2^40 }.
//     Multiplies and shifts only, with the reciprocals taken before the sums arrive.
//  2. The exact stage of avtp_exact.cuh takes the partition of the images into
//     clamped-low, free and clamped-high that this shift implies, checks it in exact
//     rational arithmetic (searching the breakpoints exactly when it does not hold),
//     and computes the kept masses x_i, their floors and the largest-remainder
//     rounding exactly. The budgets are therefore those of the plain rule, whatever
//     the grid's rounding.
//
// G is continuous, non-decreasing and linear between the breakpoints
// R_min - R_i and R_max - R_i, so for up to kBreakpointImages images the grid's lambda
// is found at the breakpoints: evaluate G at every breakpoint, take the two that bracket
// the target and solve the linear piece between them with one integer division.
// Beyond that a 32-way multisection gives the same lambda.
//
// Everything is warp-synchronous (shuffles and __syncwarp only): on this part a
// block-wide barrier or a dependent fp64 operation or division costs far more than
// the arithmetic.
#pragma once

#include "avtp_exact.cuh"

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
  float r_base_f;  // the request's keep ratio
  int64_t Rb;    // rint(r_base * 2^40)
  int64_t coef;  // alpha (additive) or r_base * alpha (relative) is coef * 2^-shift on the grid
  int shift;
  int relative;
};

__device__ __forceinline__ RatioRule make_ratio_rule(float r_base, float alpha, int relative) {
  RatioRule q;
  q.r_base_f = r_base;
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

// The exact stage for a request whose images sit in sm (S, n, R on the grid) and whose
// grid shift is lam: the width that holds the rule's products, see avtp_exact.cuh.
__device__ __forceinline__ int exact_stage(const WarpAllocSmem& sm, int m, int64_t B, int32_t N, int64_t T,
                                           float r_base_f, float alpha_f, float r_min_f, float r_max_f, int relative,
                                           int64_t lam, int64_t Rmin, int64_t Rmax) {
  const ExactRule q = make_exact_rule(B, N, T, r_base_f, alpha_f, r_min_f, r_max_f, relative);
  if (relative && q.mode == kExactGeneral) return exact_budgets<I256>(sm, m, q, lam, Rmin, Rmax);
  return exact_budgets<i128>(sm, m, q, lam, Rmin, Rmax);
}

// All 32 lanes call with identical scalars. sm.S[j] = S_j and sm.n[j] = n_j for j < m on
// entry; the budgets are left in sm.K. Returns AVTP_OK, AVTP_ERR_DEVICE_INPUT for a sum
// beyond n_j * 2^42, or AVTP_ERR_RANGE if the rounding loop did not converge (never
// expected).
static __device__ __noinline__ int warp_allocate(const WarpAllocSmem& sm, int m, int64_t B, int32_t N, float r_base_f,
                                                 float alpha_f, float r_min_f, float r_max_f, int relative) {
  const int lane = threadIdx.x & 31;
  const int64_t Rmin = ratio_grid(r_min_f), Rmax = ratio_grid(r_max_f);
  // ---- ratios on the grid
  int64_t part = 0;
  bool bad = false;
  for (int j = lane; j < m; j += 32) {
    const int64_t S = sm.S[j], lim = static_cast<int64_t>(sm.n[j]) << kSumMagnitudeBits;
    bad |= S > lim || S < -lim;
    part += S;
  }
  if (__any_sync(0xffffffffu, bad)) return AVTP_ERR_DEVICE_INPUT;
  const int64_t T = warp_sum(part);
  const int64_t avg = grid_mean(T, recip62(N));
  const int64_t inv_avg = (relative && avg != 0) ? recip62(avg > 0 ? avg : -avg) : 0;
  const RatioRule rule = make_ratio_rule(r_base_f, alpha_f, relative);
  int64_t mx = INT64_MIN, mn = INT64_MAX;
  for (int j = lane; j < m; j += 32) {
    const int64_t g = grid_ratio(rule, grid_mean(sm.S[j], recip62(sm.n[j])), avg, inv_avg);
    sm.R[j] = g;
    mx = g > mx ? g : mx;
    mn = g < mn ? g : mn;
  }
  mx = warp_max64(mx);
  mn = warp_min64(mn);
  __syncwarp();

  // ---- the grid's water-fill shift
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

  return exact_stage(sm, m, B, N, T, r_base_f, alpha_f, r_min_f, r_max_f, relative, lam, Rmin, Rmax);
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

// ---------------------------------------------------------------- the register path's exact stage
// For requests of at most 32 images, lane j owning image j: the arithmetic of
// exact_budgets (avtp_exact.cuh) held in registers, with no shared memory and no call on
// the common path. Every kept mass is written as x_i = X_i / (2^64 Q) with integers
// X_i >= 0 and Q >= 1 common to the request:
//   every image at r_min:   X_i = n_i m 2^32,  Q = 1
//   every image at r_max:   X_i = n_i M 2^32,  Q = 1
//   one common ratio:       X_i = n_i B 2^64,  Q = N
//   general:                X_i of avtp_exact.cuh (its E is 2^64 Q), Q = N_F for the
//                           additive rule and |sum S| N_F for the relative one,
// so k_i = floor((X_i >> 64) / Q), and the remainders order as the pairs
// ((X_i >> 64) mod Q, X_i mod 2^64). Returns kExactFallback when the grid's partition
// does not verify or the rounding would give an image more than one token; the caller
// then runs the general stage.
constexpr int kExactFallback = -1;

__device__ __forceinline__ unsigned bit_length_u128(u128 v) {
  const uint64_t hi = static_cast<uint64_t>(v >> 64), lo = static_cast<uint64_t>(v);
  return hi ? 128u - __clzll(static_cast<long long>(hi)) : (lo ? 64u - __clzll(static_cast<long long>(lo)) : 0u);
}

__device__ __forceinline__ float u128_to_float(u128 v) {
  return __ull2float_rn(static_cast<uint64_t>(v >> 64)) * 18446744073709551616.f +
         __ull2float_rn(static_cast<uint64_t>(v));
}

// cls: this lane's image in the partition to check (kClsFree, kClsLow or kClsHigh);
// all_free: every image is free, which needs no class sums.
template <bool kRel>
__device__ __forceinline__ int exact32(bool has, int64_t S, int64_t n, int cls, bool all_free, int64_t B, int64_t N,
                                       int64_t T, int64_t Rb, int64_t Aa, int64_t mq, int64_t Mq, int32_t* k_out) {
  const int lane = threadIdx.x & 31;
  if (!has) { S = 0; n = 0; }
  u128 Xh = 0, Q = 1;  // X_i >> 64, and the request's Q
  uint64_t Xl = 0;     // X_i mod 2^64
  if ((B << 32) <= N * mq || (B << 32) >= N * Mq) {
    const u128 X = static_cast<u128>(n * ((B << 32) <= N * mq ? mq : Mq)) << 32;
    Xh = X >> 64;
    Xl = static_cast<uint64_t>(X);
  } else if (Aa == 0 || (kRel && (T == 0 || Rb == 0))) {
    Xh = static_cast<u128>(n * B);
    Q = static_cast<u128>(N);
  } else {
    // ---- the partition, checked exactly
    if (!has) cls = kClsFree;
    const int64_t sgn = (kRel && T < 0) ? -1 : 1;
    const int64_t y = sgn * S;
    int64_t NL = 0, NH = 0, NF = N, YF = sgn * T;
    if (!all_free) {
      NL = warp_sum(cls == kClsLow ? n : int64_t(0));
      NH = warp_sum(cls == kClsHigh ? n : int64_t(0));
      NF = warp_sum(cls == kClsFree ? n : int64_t(0));
      YF = warp_sum(cls == kClsFree ? y : int64_t(0));
    }
    if (NF == 0) return kExactFallback;
    const int64_t W = (B << 32) - mq * NL - Mq * NH;
    const i128 Dd = static_cast<i128>(y) * NF - static_cast<i128>(n) * YF;
    const i128 nlo = static_cast<i128>(n) * mq * NF, nhi = static_cast<i128>(n) * Mq * NF;
    bool ok;
    if (!kRel) {
      // Kn = alpha 2^32, Kd = 2^32: every product below 2^127
      const i128 v = static_cast<i128>(Aa) * Dd + (static_cast<i128>(n) * W << 32);
      const i128 lo = nlo << 32, hi = nhi << 32;
      ok = cls == kClsLow ? v <= lo : (cls == kClsHigh ? v >= hi : (v >= lo && v <= hi));
      const u128 X = static_cast<u128>(cls == kClsLow ? lo : (cls == kClsHigh ? hi : v));
      Xh = X >> 64;
      Xl = static_cast<uint64_t>(X);
      Q = static_cast<u128>(NF);
    } else {
      // Kn = (r_base 2^32)(alpha 2^32) N, Kd = |sum S| 2^32: 256-bit products
      const i128 Kn = static_cast<i128>(Rb) * Aa * N;
      const i128 Kd = static_cast<i128>(T < 0 ? -T : T) << 32;
      const I256 v = i256_add(i256_mul(Kn, Dd), i256_mul(Kd, static_cast<i128>(n) * W));
      const I256 lo = i256_mul(Kd, nlo), hi = i256_mul(Kd, nhi);
      ok = cls == kClsLow ? i256_cmp(v, lo) <= 0
                          : (cls == kClsHigh ? i256_cmp(v, hi) >= 0 : (i256_cmp(v, lo) >= 0 && i256_cmp(v, hi) <= 0));
      const I256& X = cls == kClsLow ? lo : (cls == kClsHigh ? hi : v);
      Xh = (static_cast<u128>(X.w[2]) << 64) | X.w[1];  // X < 2^192: the top word is 0
      Xl = X.w[0];
      Q = static_cast<u128>(T < 0 ? -T : T) * static_cast<u128>(NF);
    }
    if (!__all_sync(0xffffffffu, !has || ok)) return kExactFallback;
  }
  // ---- floor and remainder: a float quotient, then an exact correction
  uint32_t q = 0;
  if (Xh != 0) {
    // within a few units of the true quotient (below 2^22 + 1), which the loops correct
    const float qf = __fdividef(u128_to_float(Xh), u128_to_float(Q));
    q = qf < 4194304.f ? static_cast<uint32_t>(qf) : 4194304u;
  }
  i128 r = static_cast<i128>(Xh) - static_cast<i128>(Q) * q;
#pragma unroll 1
  for (int it = 0; it < 4 && r < 0; ++it) { --q; r += static_cast<i128>(Q); }
#pragma unroll 1
  for (int it = 0; it < 4 && r >= static_cast<i128>(Q); ++it) { ++q; r -= static_cast<i128>(Q); }
  const u128 rem_hi = static_cast<u128>(r);
  int32_t K = has ? static_cast<int32_t>(q < static_cast<uint32_t>(n) ? q : static_cast<uint32_t>(n)) : 0;
  // ---- largest remainder: one token for each of the |D| images served first
  // (0 <= K and the sum of the K below 2^31, so one 32-bit warp reduction gives it)
  const int64_t D = B - static_cast<int64_t>(__reduce_add_sync(0xffffffffu, static_cast<uint32_t>(K)));
  if (D != 0) {
    const bool up = D > 0;
    const int need = static_cast<int>(up ? D : -D);
    const bool elig = has && (up ? K < n : K > 0);
    unsigned cand = __ballot_sync(0xffffffffu, elig);
    if (__popc(cand) < need) return kExactFallback;
    // 59-bit prefix of the remainder (rem_hi 2^64 + Xl < 2^(bq + 64)); its order is the
    // order of the remainders, up to ties among equal prefixes
    const unsigned s = bit_length_u128(Q) + 5u;
    const uint64_t prefix = s >= 64 ? static_cast<uint64_t>(rem_hi >> (s - 64))
                                    : static_cast<uint64_t>((rem_hi << (64 - s)) | (Xl >> s));
    const uint64_t kPrefixMask = (uint64_t(1) << 59) - 1;
    // adding: the largest remainders first; removing: the smallest
    const uint64_t pkey = !elig ? 0ull : (up ? prefix : kPrefixMask - prefix);
    // the `need` largest keys by a bitwise radix select with ballots, from the highest bit
    // any candidate sets: a bit splits the candidates into ones (served first) and zeros
    int left = need;
    unsigned served = 0;
    const unsigned hi_or = __reduce_or_sync(0xffffffffu, static_cast<uint32_t>(pkey >> 32));
    const unsigned lo_or = __reduce_or_sync(0xffffffffu, static_cast<uint32_t>(pkey));
    int bit = hi_or ? 63 - __clz(hi_or) : (lo_or ? 31 - __clz(lo_or) : -1);
#pragma unroll 1
    for (; bit >= 0 && __popc(cand) > left; --bit) {
      const unsigned ones = __ballot_sync(0xffffffffu, (pkey >> bit) & 1ull) & cand;
      const int c = __popc(ones);
      if (c >= left) {
        cand = ones;
      } else {
        served |= ones;
        left -= c;
        cand &= ~ones;
      }
    }
    if (__popc(cand) > left) {
      // the cut falls among candidates with equal prefixes: order those exactly, ties to the
      // lower image when adding and to the higher one when removing
      const bool in_group = (cand >> lane) & 1u;
      const uint64_t rh1 = static_cast<uint64_t>(rem_hi >> 64), rh0 = static_cast<uint64_t>(rem_hi);
      int rank = 0;
      for (unsigned g = cand; g != 0; g &= g - 1) {
        const int l = __ffs(g) - 1;
        const uint64_t a1 = __shfl_sync(0xffffffffu, rh1, l), a0 = __shfl_sync(0xffffffffu, rh0, l);
        const uint64_t al = __shfl_sync(0xffffffffu, Xl, l);
        int c = a1 != rh1 ? (a1 > rh1 ? 1 : -1) : (a0 != rh0 ? (a0 > rh0 ? 1 : -1) : (al != Xl ? (al > Xl ? 1 : -1) : 0));
        if (!up) c = -c;  // removing: the smaller remainder first
        rank += (l != lane && (c > 0 || (c == 0 && (up ? l < lane : l > lane)))) ? 1 : 0;
      }
      served |= __ballot_sync(0xffffffffu, in_group && rank < left);
    } else {
      served |= cand;
    }
    if ((served >> lane) & 1u) K += up ? 1 : -1;
  }
  *k_out = K;
  return AVTP_OK;
}

// A clamp binds: the grid's shift proposes the partition, checked exactly; the general
// stage when that does not settle it. Out of line: fetched only when it runs.
// The grid's shift: without clamps G is linear with slope N, so the smallest solution is
// lambda0 = ceil((B * 2^40 - sum n_i R_i) / N); when no clamp binds at lambda0 - 1 or
// lambda0, G is that line on [lambda0 - 1, lambda0] and lambda0 is exact. Otherwise the
// breakpoints decide.
static __device__ __noinline__ int warp_allocate32_clamped(const WarpAllocSmem& sm, int m, int64_t S, int32_t n,
                                                           int64_t inv_n, int64_t B, int32_t N, int64_t inv_N,
                                                           int64_t T, const RatioRule& rule, float alpha_f,
                                                           float r_min_f, float r_max_f, int64_t Rb, int64_t Aa,
                                                           int64_t mq, int64_t Mq, int32_t* k_out) {
  const int lane = threadIdx.x & 31;
  const bool has = lane < m;
  const int64_t Rmin = ratio_grid(r_min_f), Rmax = ratio_grid(r_max_f);
  // ---- ratios on the grid
  const int64_t avg = grid_mean(T, inv_N);
  const int64_t inv_avg = (rule.relative && avg != 0) ? recip62(avg > 0 ? avg : -avg) : 0;
  const int64_t R = has ? grid_ratio(rule, grid_mean(S, inv_n), avg, inv_avg) : 0;
  const int64_t mx = warp_max64(has ? R : INT64_MIN);
  const int64_t mn = warp_min64(has ? R : INT64_MAX);
  const int64_t target = B << kRatioFracBits;
  const int64_t nl = has ? n : 0;

  // ---- the grid's water-fill shift
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

  // ---- the exact stage on the grid's partition, in registers
  const int64_t g = R + lam;
  const int cls = g <= Rmin ? kClsLow : (g >= Rmax ? kClsHigh : kClsFree);
  int32_t K = 0;
  int err = rule.relative ? exact32<true>(has, S, n, cls, false, B, N, T, Rb, Aa, mq, Mq, &K)
                          : exact32<false>(has, S, n, cls, false, B, N, T, Rb, Aa, mq, Mq, &K);
  if (err == kExactFallback) {
    if (has) {
      sm.S[lane] = S;
      sm.n[lane] = n;
      sm.R[lane] = R;
    }
    __syncwarp();
    err = exact_stage(sm, m, B, N, T, rule.r_base_f, alpha_f, r_min_f, r_max_f, rule.relative, lam, Rmin, Rmax);
    K = has ? sm.K[lane] : 0;
    __syncwarp();
  }
  *k_out = K;
  return err;
}

// The same rule for requests of at most 32 images, held in registers: lane j owns image
// j (S_j, n_j in; its budget out). The partition with every image free (no clamp binds,
// the common case) is checked exactly first; only when it fails does the grid search for
// the shift (warp_allocate32_clamped), and only when that partition fails too does the
// general stage run on sm (32 entries). Identical results and status to warp_allocate.
// inv_n = floor(2^62 / n_j) and inv_N = floor(2^62 / N) come from the caller, which
// can take them before the sums are ready. Inlined: the fused selection kernel calls it
// from one place for both its warm-up run and its real run, and a call would put the
// caller's state on the stack.
__device__ __forceinline__ int warp_allocate32(const WarpAllocSmem& sm, int m, int64_t S, int32_t n, int64_t inv_n,
                                                   int64_t B, int32_t N, int64_t inv_N, const RatioRule& rule,
                                                   float alpha_f, float r_min_f, float r_max_f, int32_t* k_out) {
  const int lane = threadIdx.x & 31;
  const bool has = lane < m;
  const int64_t lim = static_cast<int64_t>(n) << kSumMagnitudeBits;
  if (__any_sync(0xffffffffu, has && (S > lim || S < -lim))) return AVTP_ERR_DEVICE_INPUT;
  const int64_t T = warp_sum(has ? S : int64_t(0));
  const int64_t Rb = units32(rule.r_base_f), Aa = units32(alpha_f), mq = units32(r_min_f), Mq = units32(r_max_f);
  int32_t K = 0;
  // ---- first the partition of the common case, no clamp binding: no search needed
  int err = rule.relative ? exact32<true>(has, S, n, kClsFree, true, B, N, T, Rb, Aa, mq, Mq, &K)
                          : exact32<false>(has, S, n, kClsFree, true, B, N, T, Rb, Aa, mq, Mq, &K);
  if (err != kExactFallback) {
    *k_out = K;
    return err;
  }
  return warp_allocate32_clamped(sm, m, S, n, inv_n, B, N, inv_N, T, rule, alpha_f, r_min_f, r_max_f, Rb, Aa, mq,
                                 Mq, k_out);
}

}  // namespace avtp
