// Exact rational arithmetic of the budget rule (paper §3.3.3 adaptive keep ratio,
// App. A.2 clamps), run by ONE WARP per request after the integer grid of
// avtp_alloc.cuh has proposed a shift.
//
// The rule, with every quantity an exact rational:
//   Ibar_i = S_i / (2^32 n_i),  Ibar_avg = sum S / (2^32 N)            (token-weighted)
//   additive: r_i = r_base + alpha (Ibar_i - Ibar_avg)
//   relative: r_i = r_base (1 + alpha (Ibar_i / Ibar_avg - 1))         (r_base if Ibar_avg = 0)
//   lambda:   sum_i n_i clamp(r_i + lambda, r_min, r_max) = B
//   x_i = n_i clamp(r_i + lambda, r_min, r_max); k_i = floor(x_i), then largest remainder.
// A shift common to every ratio is absorbed by lambda, so only the part of r_i that
// differs between images matters: w_i = kappa * y_i / n_i with
//   additive: kappa = alpha / 2^32,                 y_i = S_i
//   relative: kappa = r_base alpha N / |sum S|,      y_i = sign(sum S) S_i
// kappa > 0 is held as Kn / (Kd 2^32) with integers Kn, Kd. For a partition of the
// images into clamped-low L, free F and clamped-high H (with N_F > 0),
//   x_i (i in F) = [kappa (y_i N_F - n_i Y_F) + n_i W / 2^32] / N_F,
//   W = B 2^32 - m N_L - M N_H,   Y_F = sum_F y_j,
// where r_min = m / 2^32 and r_max = M / 2^32. Over the common denominator
// E = Kd 2^32 N_F every x_i is the integer X_i = x_i E:
//   X_i = Kn (y_i N_F - n_i Y_F) + Kd n_i W    (free),
//   X_i = Kd n_i m N_F (low),   X_i = Kd n_i M N_F (high).
// A partition is the right one exactly when every free X_i lies within
// [Kd n_i m N_F, Kd n_i M N_F], every low one's free value at or below the lower
// end and every high one's at or above the upper end; then G(lambda) = B holds by
// construction and the X_i are the kept masses, with no rounding anywhere.
//
// Sizes. Parameters are multiples of 2^-32 (alpha in [0, 1024], ratios in [0, 1]),
// |S_i| <= n_i 2^42 and N <= 2^20. The additive rule has Kn = alpha 2^32 <= 2^42 and
// Kd = 2^32, so every product stays below 2^127: 128-bit integers suffice. The
// relative rule has Kn = (r_base 2^32)(alpha 2^32) N <= 2^94 and Kd = 2^32 |sum S| <= 2^94,
// and products reach about 2^178: it uses the 256-bit type below.
//
// The partition comes from the grid's shift. When it does not verify (a breakpoint
// within the grid's rounding of the solution, or every image clamped), an exact search
// over the breakpoints r_min - w_i and r_max - w_i takes over: each round evaluates
// G >= B at one breakpoint in exact arithmetic and discards every breakpoint on the
// wrong side of it, until the solution's open interval holds none.
#pragma once

#include "avtp_internal.cuh"

namespace avtp {

typedef __int128 i128;
typedef unsigned __int128 u128;

// ---------------------------------------------------------------- 256-bit integers
// Two's complement, w[0] least significant.
struct I256 {
  uint64_t w[4];
};

__device__ __forceinline__ I256 i256_of(i128 x) {
  const u128 u = static_cast<u128>(x);
  const uint64_t s = x < 0 ? ~0ull : 0ull;
  return I256{{static_cast<uint64_t>(u), static_cast<uint64_t>(u >> 64), s, s}};
}

__device__ __forceinline__ I256 i256_add(const I256& a, const I256& b) {
  I256 r;
  uint64_t c = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const u128 s = static_cast<u128>(a.w[k]) + b.w[k] + c;
    r.w[k] = static_cast<uint64_t>(s);
    c = static_cast<uint64_t>(s >> 64);
  }
  return r;
}

__device__ __forceinline__ I256 i256_neg(const I256& a) {
  I256 r;
  uint64_t c = 1;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const u128 s = static_cast<u128>(~a.w[k]) + c;
    r.w[k] = static_cast<uint64_t>(s);
    c = static_cast<uint64_t>(s >> 64);
  }
  return r;
}

__device__ __forceinline__ I256 i256_sub(const I256& a, const I256& b) { return i256_add(a, i256_neg(b)); }

__device__ __forceinline__ int i256_cmp(const I256& a, const I256& b) {
  if (a.w[3] != b.w[3]) return static_cast<int64_t>(a.w[3]) < static_cast<int64_t>(b.w[3]) ? -1 : 1;
#pragma unroll
  for (int k = 2; k >= 0; --k)
    if (a.w[k] != b.w[k]) return a.w[k] < b.w[k] ? -1 : 1;
  return 0;
}

// a * b for |a|, |b| < 2^127 (the product is below 2^254).
static __device__ __noinline__ I256 i256_mul(i128 a, i128 b) {
  const bool neg = (a < 0) != (b < 0);
  const u128 ua = a < 0 ? static_cast<u128>(-a) : static_cast<u128>(a);
  const u128 ub = b < 0 ? static_cast<u128>(-b) : static_cast<u128>(b);
  const uint64_t a0 = static_cast<uint64_t>(ua), a1 = static_cast<uint64_t>(ua >> 64);
  const uint64_t b0 = static_cast<uint64_t>(ub), b1 = static_cast<uint64_t>(ub >> 64);
  const u128 p00 = static_cast<u128>(a0) * b0, p01 = static_cast<u128>(a0) * b1;
  const u128 p10 = static_cast<u128>(a1) * b0, p11 = static_cast<u128>(a1) * b1;
  I256 r;
  r.w[0] = static_cast<uint64_t>(p00);
  const u128 mid = (p00 >> 64) + static_cast<uint64_t>(p01) + static_cast<uint64_t>(p10);
  r.w[1] = static_cast<uint64_t>(mid);
  const u128 hi = (mid >> 64) + (p01 >> 64) + (p10 >> 64) + static_cast<uint64_t>(p11);
  r.w[2] = static_cast<uint64_t>(hi);
  r.w[3] = static_cast<uint64_t>(hi >> 64) + static_cast<uint64_t>(p11 >> 64);
  return neg ? i256_neg(r) : r;
}

// ---------------------------------------------------------------- the two integer widths
// Wide<i128> for the additive rule, Wide<I256> for the relative rule: the same exact
// formulas over the width that holds their products.
template <class T>
struct Wide;

template <>
struct Wide<i128> {
  typedef i128 T;
  static __device__ __forceinline__ T mul(i128 a, i128 b) { return a * b; }
  static __device__ __forceinline__ T add(T a, T b) { return a + b; }
  static __device__ __forceinline__ T sub(T a, T b) { return a - b; }
  static __device__ __forceinline__ int cmp(T a, T b) { return a < b ? -1 : (a > b ? 1 : 0); }
  static __device__ __forceinline__ bool neg(T a) { return a < 0; }
  // v * q for v >= 0 and 0 <= q < 2^32 (no overflow by the caller's bounds)
  static __device__ __forceinline__ T mul_small(T v, uint32_t q) { return v * static_cast<i128>(q); }
  // the three low 64-bit words of v >= 0 (v < 2^192)
  static __device__ __forceinline__ void words(T v, uint64_t* w) {
    const u128 u = static_cast<u128>(v);
    w[0] = static_cast<uint64_t>(u);
    w[1] = static_cast<uint64_t>(u >> 64);
    w[2] = 0;
  }
};

template <>
struct Wide<I256> {
  typedef I256 T;
  static __device__ __forceinline__ T mul(i128 a, i128 b) { return i256_mul(a, b); }
  static __device__ __forceinline__ T add(const T& a, const T& b) { return i256_add(a, b); }
  static __device__ __forceinline__ T sub(const T& a, const T& b) { return i256_sub(a, b); }
  static __device__ __forceinline__ int cmp(const T& a, const T& b) { return i256_cmp(a, b); }
  static __device__ __forceinline__ bool neg(const T& a) { return static_cast<int64_t>(a.w[3]) < 0; }
  static __device__ __forceinline__ T mul_small(const T& v, uint32_t q) {
    I256 r;
    uint64_t c = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const u128 p = static_cast<u128>(v.w[k]) * q + c;
      r.w[k] = static_cast<uint64_t>(p);
      c = static_cast<uint64_t>(p >> 64);
    }
    return r;
  }
  static __device__ __forceinline__ void words(const T& v, uint64_t* w) {
    w[0] = v.w[0];
    w[1] = v.w[1];
    w[2] = v.w[2];
  }
};

// Approximate value of v >= 0 (v < 2^192 given as three words) times 2^-shift, as a
// float: used only for a first guess of a quotient that is then corrected exactly.
__device__ __forceinline__ float words_to_float_scaled(const uint64_t* w, int shift) {
  // take the 64 bits starting at `shift` (shift may be 0..191)
  const int q = shift >> 6, r = shift & 63;
  const uint64_t lo = q < 3 ? w[q] : 0;
  const uint64_t mid = q + 1 < 3 ? w[q + 1] : 0;
  const uint64_t hi = q + 2 < 3 ? w[q + 2] : 0;
  const uint64_t x0 = r ? (lo >> r) | (mid << (64 - r)) : lo;
  const uint64_t x1 = r ? (mid >> r) | (hi << (64 - r)) : mid;
  return __ull2float_rn(x1) * 18446744073709551616.f + __ull2float_rn(x0);
}

__device__ __forceinline__ int words_bit_length(const uint64_t* w) {
  if (w[2]) return 128 + 64 - __clzll(static_cast<long long>(w[2]));
  if (w[1]) return 64 + 64 - __clzll(static_cast<long long>(w[1]));
  return w[0] ? 64 - __clzll(static_cast<long long>(w[0])) : 0;
}

// floor(X / E) and X mod E for 0 <= X < 2^21 E and E > 0. A float quotient of the top
// bits is within one of the answer; one or two exact corrections finish it.
template <class T>
__device__ __forceinline__ uint32_t exact_floor_div(const T& X, const T& E, int e_bits, T* rem) {
  typedef Wide<T> O;
  uint64_t xw[3], ew[3];
  O::words(X, xw);
  O::words(E, ew);
  const int shift = e_bits > 62 ? e_bits - 62 : 0;
  const float qf = words_to_float_scaled(xw, shift) / words_to_float_scaled(ew, shift);
  uint32_t q = qf > 0.f ? static_cast<uint32_t>(qf) : 0u;
  if (q > (1u << 22)) q = 1u << 22;
  T r = O::sub(X, O::mul_small(E, q));
#pragma unroll 1
  for (int it = 0; it < 4 && O::neg(r); ++it) {
    --q;
    r = O::add(r, E);
  }
#pragma unroll 1
  for (int it = 0; it < 4 && O::cmp(r, E) >= 0; ++it) {
    ++q;
    r = O::sub(r, E);
  }
  *rem = r;
  return q;
}

// ---------------------------------------------------------------- the request's constants
enum { kExactAllLow = 0, kExactAllHigh = 1, kExactUniform = 2, kExactGeneral = 3 };
enum { kClsFree = 0, kClsLow = 1, kClsHigh = 2 };

struct ExactRule {
  int mode;     // one of the kExact* values
  int relative;
  int64_t B;    // the request's global budget
  int64_t N;    // its visual tokens
  int64_t m, M; // r_min, r_max in units of 2^-32
  int64_t sgn;  // y_i = sgn * S_i
  i128 Kn, Kd;  // kappa = Kn / (Kd 2^32) > 0 (general mode)
};

// v * 2^32 for an fp32 v >= 0 that is a multiple of 2^-32 (checked before any launch).
__device__ __forceinline__ int64_t units32(float v) {
  const uint32_t b = __float_as_uint(v);
  const int e8 = (b >> 23) & 0xff;
  if (e8 == 0) return 0;  // zero (subnormals are not multiples of 2^-32)
  const int64_t mant = (b & 0x7fffff) | 0x800000;
  const int sh = e8 - 150 + 32;  // v * 2^32 = mant * 2^sh
  return sh >= 0 ? (mant << sh) : (mant >> -sh);
}

__device__ __forceinline__ ExactRule make_exact_rule(int64_t B, int64_t N, int64_t T, float r_base, float alpha,
                                                     float r_min, float r_max, int relative) {
  ExactRule q;
  q.relative = relative;
  q.B = B;
  q.N = N;
  q.m = units32(r_min);
  q.M = units32(r_max);
  q.sgn = 1;
  q.Kn = 0;
  q.Kd = 1;
  const int64_t Aa = units32(alpha), Rb = units32(r_base);
  if ((B << 32) <= N * q.m) {
    q.mode = kExactAllLow;
  } else if ((B << 32) >= N * q.M) {
    q.mode = kExactAllHigh;
  } else if (Aa == 0 || (relative && (T == 0 || Rb == 0))) {
    q.mode = kExactUniform;
  } else {
    q.mode = kExactGeneral;
    if (!relative) {
      q.Kn = Aa;
      q.Kd = static_cast<i128>(1) << 32;
    } else {
      q.sgn = T > 0 ? 1 : -1;
      q.Kn = static_cast<i128>(Rb) * Aa * N;
      q.Kd = static_cast<i128>(T > 0 ? T : -T) << 32;
    }
  }
  return q;
}

// ---------------------------------------------------------------- per-warp scratch
// One entry per image of the request (structure of arrays).
struct WarpAllocSmem {
  int64_t* S;     // fixed-point sums
  int64_t* R;     // ratios on the grid (the search hint)
  uint64_t* rem;  // [3][m_cap]: exact remainder X_i mod E, three 64-bit words
  int32_t* n;     // image sizes
  int32_t* K;     // budgets (and per-round decisions)
  uint8_t* cls;   // kClsFree / kClsLow / kClsHigh
  uint8_t* alive; // breakpoints still in play during the exact search (bit 0: low, bit 1: high)
  int m_cap;
};

__host__ __device__ constexpr size_t warp_alloc_smem_bytes(int m_cap) {
  return (static_cast<size_t>(m_cap) * (8 + 8 + 24 + 4 + 4 + 1 + 1) + 15) & ~static_cast<size_t>(15);
}

__device__ __forceinline__ WarpAllocSmem carve_warp_alloc(unsigned char* base, int m_cap) {
  WarpAllocSmem s;
  s.m_cap = m_cap;
  s.S = reinterpret_cast<int64_t*>(base);
  s.R = s.S + m_cap;
  s.rem = reinterpret_cast<uint64_t*>(s.R + m_cap);
  s.n = reinterpret_cast<int32_t*>(s.rem + 3 * m_cap);
  s.K = s.n + m_cap;
  s.cls = reinterpret_cast<uint8_t*>(s.K + m_cap);
  s.alive = s.cls + m_cap;
  return s;
}

// ---------------------------------------------------------------- exact pieces
struct ClassSums {
  int64_t NL, NH, NF, YF;
};

__device__ __forceinline__ ClassSums class_sums(const WarpAllocSmem& sm, int m, int64_t sgn) {
  const int lane = threadIdx.x & 31;
  int64_t nl = 0, nh = 0, nf = 0, yf = 0;
  for (int j = lane; j < m; j += 32) {
    const int c = sm.cls[j];
    const int64_t nj = sm.n[j];
    nl += c == kClsLow ? nj : 0;
    nh += c == kClsHigh ? nj : 0;
    nf += c == kClsFree ? nj : 0;
    yf += c == kClsFree ? sgn * sm.S[j] : 0;
  }
  return ClassSums{warp_sum(nl), warp_sum(nh), warp_sum(nf), warp_sum(yf)};
}

// X_i of image j under the partition summed in s (see the head of this file).
template <class T>
__device__ __forceinline__ T exact_mass(const ExactRule& q, const ClassSums& s, int64_t y, int64_t n, int cls) {
  typedef Wide<T> O;
  if (cls == kClsLow) return O::mul(q.Kd, static_cast<i128>(n) * q.m * s.NF);
  if (cls == kClsHigh) return O::mul(q.Kd, static_cast<i128>(n) * q.M * s.NF);
  const int64_t W = (q.B << 32) - q.m * s.NL - q.M * s.NH;
  const i128 D = static_cast<i128>(y) * s.NF - static_cast<i128>(n) * s.YF;
  return O::add(O::mul(q.Kn, D), O::mul(q.Kd, static_cast<i128>(n) * W));
}

// Does image j's free value agree with its class? (the partition is the solution when
// every image's does)
template <class T>
__device__ __forceinline__ bool exact_class_holds(const ExactRule& q, const ClassSums& s, int64_t y, int64_t n,
                                                  int cls) {
  typedef Wide<T> O;
  const T v = exact_mass<T>(q, s, y, n, kClsFree);
  const T lo = exact_mass<T>(q, s, y, n, kClsLow);
  const T hi = exact_mass<T>(q, s, y, n, kClsHigh);
  if (cls == kClsLow) return O::cmp(v, lo) <= 0;
  if (cls == kClsHigh) return O::cmp(v, hi) >= 0;
  return O::cmp(v, lo) >= 0 && O::cmp(v, hi) <= 0;
}

// Sign of bp(ta, a) - bp(tb, b), where bp(0, j) = r_min - w_j and bp(1, j) = r_max - w_j
// are image j's breakpoints: multiplied by 2^32 Kd n_a n_b > 0 the difference is
// dt Kd n_a n_b - Kn (y_a n_b - y_b n_a), dt = (t_a ? M : m) - (t_b ? M : m).
template <class T>
__device__ __noinline__ int bp_cmp(const ExactRule& q, int ta, int64_t ya, int64_t na, int tb, int64_t yb,
                                   int64_t nb) {
  typedef Wide<T> O;
  const i128 cross = static_cast<i128>(ya) * nb - static_cast<i128>(yb) * na;
  const int64_t dt = (ta ? q.M : q.m) - (tb ? q.M : q.m);
  if (dt == 0) return cross > 0 ? -1 : (cross < 0 ? 1 : 0);
  return O::cmp(O::mul(static_cast<i128>(dt) * na * nb, q.Kd), O::mul(q.Kn, cross));
}

// Is G(bp(tp, p)) >= B, given the class sums at that breakpoint?
//   G = (m N_L + M N_H + t_p N_F) / 2^32 + kappa (Y_F n_p - N_F y_p) / n_p; times 2^32 Kd n_p:
//   Kn (Y_F n_p - N_F y_p) >= Kd n_p (B 2^32 - m N_L - M N_H - t_p N_F).
template <class T>
__device__ __noinline__ bool g_reaches_budget(const ExactRule& q, const ClassSums& s, int tp, int64_t yp,
                                              int64_t np) {
  typedef Wide<T> O;
  const i128 lhs = static_cast<i128>(s.YF) * np - static_cast<i128>(s.NF) * yp;
  const int64_t w = (q.B << 32) - q.m * s.NL - q.M * s.NH - (tp ? q.M : q.m) * s.NF;
  return O::cmp(O::mul(q.Kn, lhs), O::mul(q.Kd, static_cast<i128>(np) * w)) >= 0;
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t u = __shfl_xor_sync(0xffffffffu, v, o);
    v = u > v ? u : v;
  }
  return v;
}

// 32-bit mix of (breakpoint, round) for the search's pivot choice.
__device__ __forceinline__ uint32_t pivot_hash(uint32_t c, uint32_t round) {
  uint32_t h = c * 0x9E3779B1u ^ (round + 0x7F4A7C15u) * 0x85EBCA77u;
  h ^= h >> 15;
  h *= 0x2C1B3C6Du;
  h ^= h >> 12;
  return h;
}

// Exact search of the solution's partition (see the head of this file). Writes sm.cls.
// The grid's shift lam_grid (with the grid ratios sm.R and the grid clamps) orders the
// first two pivots: the breakpoints just below and just above it.
template <class T>
__device__ __noinline__ void exact_search(const WarpAllocSmem& sm, int m, const ExactRule& q, int64_t lam_grid,
                                          int64_t Rmin, int64_t Rmax) {
  const int lane = threadIdx.x & 31;
  const bool one_clamp = q.m == q.M;  // both breakpoints of an image coincide
  for (int j = lane; j < m; j += 32) sm.alive[j] = one_clamp ? 1 : 3;
  __syncwarp();
  int lo_t = -1, lo_j = -1, hi_t = -1, hi_j = -1;  // bracketing breakpoints found so far (-1: none)
#pragma unroll 1
  for (int round = 0; round < 2 * kMaxImagesPerRequest + 2; ++round) {
    // ---- pivot: an alive breakpoint chosen by a 64-bit key, largest key wins
    // key bits: 63 alive, 62 preferred in this iteration, 61..14 order value, 13..0 breakpoint index
    uint64_t best = 0;
    for (int j = lane; j < m; j += 32) {
      const int al = sm.alive[j];
      for (int t = 0; t < 2; ++t) {
        if (!((al >> t) & 1)) continue;
        const int64_t g = (t ? Rmax : Rmin) - sm.R[j];  // the breakpoint on the grid
        const uint64_t u = static_cast<uint64_t>(g) ^ (uint64_t(1) << 63);  // order-preserving
        uint64_t pref, val;
        if (round == 0) { pref = g <= lam_grid; val = u >> 16; }        // the highest at or below the grid shift
        else if (round == 1) { pref = g > lam_grid; val = ~u >> 16; }   // the lowest above it
        else { pref = 1; val = pivot_hash(static_cast<uint32_t>(2 * j + t), round); }
        const uint64_t key = (uint64_t(1) << 63) | (pref << 62) | ((val & ((uint64_t(1) << 48) - 1)) << 14) |
                             static_cast<uint64_t>(2 * j + t);
        best = key > best ? key : best;
      }
    }
    best = warp_max_u64(best);
    if (best == 0) break;  // nothing alive: the bracket is found
    const int pc = static_cast<int>(best & 0x3fff);
    const int pt = pc & 1, pj = pc >> 1;
    const int64_t py = q.sgn * sm.S[pj], pn = sm.n[pj];
    // ---- G at the pivot
    for (int j = lane; j < m; j += 32) {
      const int64_t y = q.sgn * sm.S[j], n = sm.n[j];
      int c = kClsFree;
      if (bp_cmp<T>(q, pt, py, pn, 0, y, n) <= 0) c = kClsLow;
      else if (bp_cmp<T>(q, pt, py, pn, 1, y, n) >= 0) c = kClsHigh;
      sm.cls[j] = static_cast<uint8_t>(c);
    }
    __syncwarp();
    const ClassSums s = class_sums(sm, m, q.sgn);
    const bool reach = g_reaches_budget<T>(q, s, pt, py, pn);
    if (reach) { hi_t = pt; hi_j = pj; } else { lo_t = pt; lo_j = pj; }
    // ---- discard the breakpoints on the pivot's side (the pivot among them)
    for (int j = lane; j < m; j += 32) {
      int al = sm.alive[j];
      const int64_t y = q.sgn * sm.S[j], n = sm.n[j];
      for (int t = 0; t < 2; ++t) {
        if (!((al >> t) & 1)) continue;
        const int c = bp_cmp<T>(q, t, y, n, pt, py, pn);
        if (reach ? c >= 0 : c <= 0) al &= ~(1 << t);
      }
      sm.alive[j] = static_cast<uint8_t>(al);
    }
    __syncwarp();
  }
  // ---- the partition on the open interval between the bracketing breakpoints
  const int64_t hy = hi_j >= 0 ? q.sgn * sm.S[hi_j] : 0, hn = hi_j >= 0 ? sm.n[hi_j] : 1;
  const int64_t ly = lo_j >= 0 ? q.sgn * sm.S[lo_j] : 0, ln = lo_j >= 0 ? sm.n[lo_j] : 1;
  for (int j = lane; j < m; j += 32) {
    const int64_t y = q.sgn * sm.S[j], n = sm.n[j];
    int c = kClsFree;
    if (hi_j >= 0 && bp_cmp<T>(q, 0, y, n, hi_t, hy, hn) >= 0) c = kClsLow;
    else if (lo_j >= 0 && bp_cmp<T>(q, 1, y, n, lo_t, ly, ln) <= 0) c = kClsHigh;
    sm.cls[j] = static_cast<uint8_t>(c);
  }
  __syncwarp();
}

// Remainder order for largest remainder: is image l served before image j?
// Adding (up): larger remainder first, ties to the lower index. Removing: smaller
// remainder first, ties to the higher index.
__device__ __forceinline__ bool served_before(const WarpAllocSmem& sm, int l, int j, bool up) {
  const int mc = sm.m_cap;
#pragma unroll
  for (int k = 2; k >= 0; --k) {
    const uint64_t a = sm.rem[k * mc + l], b = sm.rem[k * mc + j];
    if (a != b) return up ? a > b : a < b;
  }
  return up ? l < j : l > j;
}

// The exact stage. On entry sm.S, sm.n and sm.R (grid ratios) hold the request's m
// images; lam_grid is the grid's shift. Writes the budgets to sm.K. Returns AVTP_OK, or
// AVTP_ERR_RANGE should the rounding not converge (not expected).
template <class T>
__device__ __noinline__ int exact_budgets(const WarpAllocSmem& sm, int m, const ExactRule& q, int64_t lam_grid,
                                          int64_t Rmin, int64_t Rmax) {
  typedef Wide<T> O;
  const int lane = threadIdx.x & 31;
  ClassSums s{0, 0, 0, 0};
  T E;
  if (q.mode == kExactGeneral) {
    for (int j = lane; j < m; j += 32) {
      const int64_t g = sm.R[j] + lam_grid;
      sm.cls[j] = static_cast<uint8_t>(g <= Rmin ? kClsLow : (g >= Rmax ? kClsHigh : kClsFree));
    }
    __syncwarp();
    s = class_sums(sm, m, q.sgn);
    bool ok = s.NF > 0;
    if (ok) {
      for (int j = lane; j < m; j += 32) ok &= exact_class_holds<T>(q, s, q.sgn * sm.S[j], sm.n[j], sm.cls[j]);
    }
    if (!__all_sync(0xffffffffu, ok)) {
      exact_search<T>(sm, m, q, lam_grid, Rmin, Rmax);
      s = class_sums(sm, m, q.sgn);
    }
    E = O::mul(q.Kd, static_cast<i128>(s.NF) << 32);
  } else if (q.mode == kExactUniform) {
    E = O::mul(q.N, 1);
  } else {
    E = O::mul(static_cast<i128>(1) << 32, 1);
  }
  uint64_t ew[3];
  O::words(E, ew);
  const int e_bits = words_bit_length(ew);
  // ---- floors and remainders
  for (int j = lane; j < m; j += 32) {
    const int64_t n = sm.n[j];
    T X;
    if (q.mode == kExactGeneral) X = exact_mass<T>(q, s, q.sgn * sm.S[j], n, sm.cls[j]);
    else if (q.mode == kExactUniform) X = O::mul(n, q.B);
    else X = O::mul(n, q.mode == kExactAllLow ? q.m : q.M);
    T r;
    const uint32_t f = exact_floor_div<T>(X, E, e_bits, &r);
    sm.K[j] = static_cast<int32_t>(f < static_cast<uint32_t>(n) ? f : static_cast<uint32_t>(n));
    uint64_t w[3];
    O::words(r, w);
    sm.rem[j] = w[0];
    sm.rem[sm.m_cap + j] = w[1];
    sm.rem[2 * sm.m_cap + j] = w[2];
  }
  __syncwarp();
  // ---- largest remainder
#pragma unroll 1
  for (int round = 0; round < 64; ++round) {
    int64_t ks = 0;
    for (int j = lane; j < m; j += 32) ks += sm.K[j];
    const int64_t D = q.B - warp_sum(ks);
    if (D == 0) return AVTP_OK;
    const bool up = D > 0;
    // decide every image from the same snapshot of K (sm.alive is free by now), then apply
    for (int j = lane; j < m; j += 32) {
      int d = 0;
      const bool elig = up ? sm.K[j] < sm.n[j] : sm.K[j] > 0;
      if (elig) {
        int64_t rank = 0;  // eligible images served before j
        for (int l = 0; l < m; ++l) {
          const bool el = up ? sm.K[l] < sm.n[l] : sm.K[l] > 0;
          rank += (el && l != j && served_before(sm, l, j, up)) ? 1 : 0;
        }
        d = rank < (up ? D : -D) ? 1 : 0;
      }
      sm.alive[j] = static_cast<uint8_t>(d);
    }
    __syncwarp();
    for (int j = lane; j < m; j += 32) sm.K[j] += sm.alive[j] ? (up ? 1 : -1) : 0;
    __syncwarp();
  }
  return AVTP_ERR_RANGE;
}

}  // namespace avtp
