// Criterion B: text-to-visual attention mass per visual token (the per-token form of
// the attention quantity of paper §3.3.2), without materialising the attention matrix:
//   s_t = 1/(Hq*|Q_r|) * sum_h sum_{q in Q_r, pos q >= pos t} exp2(z2(h,q,t) - lse2(h,q)),
//   z2 = softmax_scale * log2(e) * q_h . k_{g(h)},  lse2 = log2 sum_{visible keys} exp2(z2).
//
// Rows: for KV group g, row o*G + j is text query o (in text order over the batch)
// with query head g*G + j. The text queries are first repacked by group into
// Qt[g][row][d] (k_attn_pack), so that both passes read them with TMA boxes. A
// request's rows are cut into blocks of 256.
//
// Pass 1, k_attn_lse (skipped when the caller supplies FlashAttention's LSE): a block
// is held as two 128-row A tiles and every key tile of 256 keys, from the request's
// first token to the block's last query, feeds two MMAs (128 x 256 x d, one per A
// tile, fp32 accumulators in TMEM), so every key byte brought to the SM serves 256
// rows. The epilogue reads accumulator 0 while the MMA of tile 1 runs and keeps an
// online (max, sum) per row; it leaves one partial per (row, CTA) behind.
// Pass 2, k_attn_mass: a block is held as the MMA B operand (N = 256 rows) and the
// tiles of 128 visual keys of every image that one of its queries follows stream
// through it as A (M = 128 keys), into two accumulators used in turn. A thread owns
// one key and sums exp2(z2 - lse2) over the rows of its column half; lse2 comes from
// the pass-1 partials of the block (merged on load) or from the supplied LSE, and is
// +inf on rows whose query precedes the key's image. The per-key sums of all blocks
// and KV groups meet in a 64-bit fixed-point accumulator (integer atomics: the result
// does not depend on their order).
// k_attn_finalize turns the accumulator into scores and the fixed-point image sums.
//
// Both passes are persistent: the flat list of (KV group, block, key step) is split
// into equal contiguous runs, one per CTA (one CTA per SM). Warps 0-7 are the epilogue
// (warp w reads TMEM lanes 32(w%4)..+31 and column half w/4 of every accumulator),
// warp 8 issues the TMA loads, warp 9 owns TMEM and issues the MMAs. TMEM holds two
// 256-column accumulators.
#include <cudaTypedefs.h>

#include "avtp_tc.cuh"

namespace avtp {
namespace {

constexpr int kM = kAttnTileM;        // 128
constexpr int kN = kAttnTileN;        // 256
constexpr int kBlk = kAttnBlockRows;  // 256
constexpr int kTmaWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kThreads = 320;
constexpr int kEpiWarps = 8;          // warps 0-7: epilogue
constexpr uint32_t kTmemCols = 2 * kN;
constexpr int kP2Stages = 4;          // key tiles in flight in pass 2
constexpr int kMassWindow = 24;       // pass-2 steps whose key masses are held in shared memory between flushes
constexpr float kLog2e = 1.4426950408889634f;
// Flag of a key whose mass is not a finite number in [0, 256] (non-finite inputs). The
// sum of its finite contributions stays below 2^62: at most 256 * 2^40 per (KV group,
// block), fewer than 2^14 of them.
constexpr unsigned long long kMassNotFinite = 1ull << 63;

static_assert(kBlk == 2 * kM && kBlk == kN, "a block is two A tiles (pass 1) and one B operand (pass 2)");

// Shared memory for head_dim d (1024-byte aligned tiles).
__host__ __device__ constexpr size_t a_bytes(int d) { return static_cast<size_t>(kM) * d * 2; }
__host__ __device__ constexpr size_t b_bytes(int d) { return static_cast<size_t>(kN) * d * 2; }
// pass 1: two A tiles (the block) + two key stages; pass 2: the block + kP2Stages key tiles
__host__ __device__ constexpr size_t lse_smem_bytes(int d) { return 1024 + 2 * a_bytes(d) + 2 * b_bytes(d); }
__host__ __device__ constexpr size_t mass_smem_bytes(int d) { return 1024 + b_bytes(d) + kP2Stages * a_bytes(d); }

struct Sync {
  uint64_t a_full[kP2Stages], a_empty[kP2Stages];
  uint64_t b_full[2], b_empty[2];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t drain;
  uint32_t tmem;
  int abort;
};

struct AttnArgs {
  const int32_t* cu;
  int R;
  const int32_t* ist;
  const int32_t* iln;
  const int32_t* icu;
  int NI;
  int64_t T;
  const int32_t* vis_cu;
  const int32_t* text_idx;
  const int32_t* text_cu;
  const int32_t* blk_cu;
  const int32_t* p1s_cu;
  const int32_t* p2t_cu;
  const int32_t* ktile_cu;
  const int32_t* meta;           // F1, C1, F2, C2
  const float* lse_rows;         // [Hkv, rows] (supplied LSE) or nullptr
  float2* p1_part;               // [Hkv * NB][256 rows][kAttnMaxChunks]
  unsigned long long* mass;      // [key tile][128] fixed point, 2^-kAttnMassFracBits
  int64_t rows;
  int G, Hkv, d;
  float c2;                      // softmax_scale * log2(e)
  DevStatus* st;
};

__device__ __forceinline__ void bar_epi() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

// Diagnostic timeline build (-DAVTP_TIMELINE): clock stamps of each pass's first CTA, per
// step s of its run. Slots: 0 the key tile's load issued (TMA thread); 1 the MMA thread at
// the step, 2 its operands and accumulators ready, 3 its MMAs issued and committed; 4 the
// step's (first) accumulator ready for epilogue warp 0, 5 the step's (last) accumulator
// released by it. Read with avtp_score_timeline().
constexpr int kAttnTlSteps = 64;
constexpr int kAttnTlSlots = 6;
#ifdef AVTP_TIMELINE
__device__ long long g_attn_tl[2][kAttnTlSteps][kAttnTlSlots];
#endif
__device__ __forceinline__ void attn_stamp(int pass, int st, int slot) {
#ifdef AVTP_TIMELINE
  if (blockIdx.x == 0 && st < kAttnTlSteps) g_attn_tl[pass][st][slot] = clock64();
#else
  (void)pass;
  (void)st;
  (void)slot;
#endif
}

// A (KV group, row block) pair: rows [R0, R1) of group g belong to request r.
struct Seg {
  int g, b, r;
  int64_t R0, R1;
};

__device__ __forceinline__ Seg seg_of(const AttnArgs& a, int g, int b) {
  Seg s;
  s.g = g;
  s.b = b;
  s.r = upper_index(a.blk_cu, a.R, b);
  s.R0 = static_cast<int64_t>(a.text_cu[s.r]) * a.G + static_cast<int64_t>(b - a.blk_cu[s.r]) * kBlk;
  s.R1 = min(s.R0 + kBlk, static_cast<int64_t>(a.text_cu[s.r + 1]) * a.G);
  return s;
}

// Walks a CTA's run of the flat list (KV group, block, entry) of a pass whose per-group
// list has F entries with prefix cu over the NB blocks. Global memory is read only
// when the walk enters a new block, so the single MMA-issuing and TMA-issuing threads
// do not wait on dependent loads between steps.
struct FlatCursor {
  int g, b, j;  // KV group, block, entry within the block
  int n;        // entries of block b
  __device__ __forceinline__ void init(int64_t f, int F, const int32_t* cu, int NB) {
    g = static_cast<int>(f / F);
    const int fl = static_cast<int>(f - static_cast<int64_t>(g) * F);
    b = upper_index(cu, NB, fl);
    j = fl - cu[b];
    n = cu[b + 1] - cu[b];
  }
  // Next entry; returns true when it lies in another block. Only called while another
  // entry exists, so the loop over empty blocks ends.
  __device__ __forceinline__ bool next(const int32_t* cu, int NB) {
    if (++j < n) return false;
    j = 0;
    do {
      if (++b == NB) {
        b = 0;
        ++g;
      }
      n = cu[b + 1] - cu[b];
    } while (n == 0);
    return true;
  }
  __device__ __forceinline__ bool last_of_block() const { return j + 1 == n; }
};

// Pass-2 key tiles of a block in order: tile j is tile jj of image i, the images of the
// block's request in order. The request's fields are read when the walk enters a block;
// the next image's fields are loaded as soon as the walk enters an image, so that their
// latency is hidden behind the steps of the current image.
struct TileCursor {
  int i, jj;           // image, tile within the image
  int kp0, nk, c0;     // first packed key, keys in the tile, first row of the block that sees it
  int tile;            // key tile over all images (row of the mass accumulator)
  int base, len, t0;   // packed position of the image's first key, its length, its first key tile
  int64_t c0_img;      // o_first(i) * G - R0
  int cu_r, text_r, vis_r0, img_end;  // the request's first token, first text ordinal, first visual ordinal, image end
  int n_ist, n_iln, n_t0, n_vis;      // image i + 1: start, length, first key tile, visual prefix after it
  __device__ __forceinline__ void prefetch(const AttnArgs& a) {
    if (i + 1 < img_end) {
      n_ist = a.ist[i + 1];
      n_iln = a.iln[i + 1];
      n_t0 = a.ktile_cu[i + 1];
      n_vis = a.vis_cu[i + 2];
    }
  }
  __device__ __forceinline__ void apply(const Seg& s, int g, int ist, int iln, int tk0, int vis1) {
    base = cu_r + ist;
    len = iln;
    t0 = tk0;
    const int64_t o_first = static_cast<int64_t>(text_r) + ist + iln - (vis1 - vis_r0);
    c0_img = o_first * g - s.R0;
  }
  __device__ __forceinline__ void fill() {
    kp0 = base + jj * kM;
    nk = min(kM, len - jj * kM);
    tile = t0 + jj;
    c0 = c0_img > 0 ? static_cast<int>(c0_img) : 0;
  }
  __device__ __forceinline__ void init(const AttnArgs& a, const Seg& s, int j) {
    const int r = s.r;
    cu_r = a.cu[r];
    text_r = a.text_cu[r];
    vis_r0 = a.vis_cu[a.icu[r]];
    img_end = a.icu[r + 1];
    const int t = a.ktile_cu[a.icu[r]] + j;
    i = upper_index(a.ktile_cu, a.NI, t);
    jj = t - a.ktile_cu[i];
    apply(s, a.G, a.ist[i], a.iln[i], a.ktile_cu[i], a.vis_cu[i + 1]);
    prefetch(a);
    fill();
  }
  __device__ __forceinline__ void next(const AttnArgs& a, const Seg& s) {
    if ((++jj) * kM >= len) {
      ++i;
      jj = 0;
      apply(s, a.G, n_ist, n_iln, n_t0, n_vis);
      prefetch(a);
    }
    fill();
  }
};

// ---------------------------------------------------------------- epilogue arithmetic
// A warp's slice of an accumulator: its 32 TMEM lanes x kHalf columns, read as 32-column
// chunks; chunk p+1 is loaded while chunk p is processed. MASKED = false is the common
// case (every column visible to every lane): straight-line code without per-chunk
// votes. The masked form handles the chunks [pb, pe) and keeps the columns c with
// lo <= c < hi (per lane in pass 1, per CTA in pass 2).
constexpr int kHalf = kN / 2;
constexpr int kChunks = kHalf / 32;

// Pass 1: online (max m, sum l) of exp2(c2 * z) over the visible columns of a row.
template <bool MASKED>
__device__ __forceinline__ void p1_slice(uint32_t taddr, int pe, int lim, float c2, float& m, float& l) {
  uint32_t ra[32], rb[32];
  auto chunk = [&](uint32_t(&r)[32], uint32_t(&nx)[32], int p) {
    if (p + 1 < pe) tc::tmem_ld32_async(taddr + (p + 1) * 32, nx);
    float v[32];
#pragma unroll
    for (int q = 0; q < 32; ++q) v[q] = __uint_as_float(r[q]);
    if (MASKED) {
#pragma unroll
      for (int q = 0; q < 32; ++q) v[q] = (p * 32 + q <= lim) ? v[q] : -INFINITY;
    }
    // max as a tree (depth 5); exact in any order
    float t16[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) t16[q] = fmaxf(v[2 * q], v[2 * q + 1]);
#pragma unroll
    for (int w = 8; w >= 1; w >>= 1) {
#pragma unroll
      for (int q = 0; q < w; ++q) t16[q] = fmaxf(t16[q], t16[q + w]);
    }
    const float mn = fmaxf(m, t16[0] * c2);
    // four partial sums (columns q mod 4), two per packed register
    const float2 cc = make_float2(c2, c2), nm = make_float2(-mn, -mn);
    float2 s01 = make_float2(0.f, 0.f), s23 = s01;
#pragma unroll
    for (int q = 0; q < 32; q += 4) {
      const float2 a01 = tc::ffma2(make_float2(v[q], v[q + 1]), cc, nm);
      const float2 a23 = tc::ffma2(make_float2(v[q + 2], v[q + 3]), cc, nm);
      s01 = tc::add2(s01, make_float2(tc::ex2(a01.x), tc::ex2(a01.y)));
      s23 = tc::add2(s23, make_float2(tc::ex2(a23.x), tc::ex2(a23.y)));
    }
    const float s0 = s01.x, s1 = s01.y, s2 = s23.x, s3 = s23.y;
    // a row with nothing visible yet keeps (-inf, 0); exp2(-inf - -inf) would be NaN
    if (mn != -INFINITY) {
      l = l * tc::ex2(m - mn) + ((s0 + s1) + (s2 + s3));
      m = mn;
    }
    if (p + 1 < pe) tc::tmem_wait(nx);
  };
  tc::tmem_ld32_async(taddr, ra);
  tc::tmem_wait(ra);
#pragma unroll
  for (int p = 0; p < kChunks; p += 2) {
    if (p < pe) chunk(ra, rb, p);
    if (p + 1 < pe) chunk(rb, ra, p + 1);
  }
}

// Pass 2: sum of exp2(c2 * z - lse2[c]) over the columns c of a key. `nlse` holds
// -lse2; a column that does not see the key carries -inf, which makes its term 0.
__device__ __forceinline__ float p2_slice(uint32_t taddr, const float* nlse, float c2) {
  uint32_t ra[32], rb[32];
  // four partial sums (columns q mod 4), two per packed register
  float2 m01 = make_float2(0.f, 0.f), m23 = m01;
  const float2 cc = make_float2(c2, c2);
  auto chunk = [&](uint32_t(&r)[32], uint32_t(&nx)[32], int p) {
    if (p + 1 < kChunks) tc::tmem_ld32_async(taddr + (p + 1) * 32, nx);
    const float4* l4 = reinterpret_cast<const float4*>(nlse + p * 32);
#pragma unroll
    for (int q4 = 0; q4 < 8; ++q4) {
      const float4 lv = l4[q4];
      const float2 a01 =
          tc::ffma2(make_float2(__uint_as_float(r[4 * q4 + 0]), __uint_as_float(r[4 * q4 + 1])), cc,
                    make_float2(lv.x, lv.y));
      const float2 a23 =
          tc::ffma2(make_float2(__uint_as_float(r[4 * q4 + 2]), __uint_as_float(r[4 * q4 + 3])), cc,
                    make_float2(lv.z, lv.w));
      m01 = tc::add2(m01, make_float2(tc::ex2(a01.x), tc::ex2(a01.y)));
      m23 = tc::add2(m23, make_float2(tc::ex2(a23.x), tc::ex2(a23.y)));
    }
    if (p + 1 < kChunks) tc::tmem_wait(nx);
  };
  tc::tmem_ld32_async(taddr, ra);
  tc::tmem_wait(ra);
#pragma unroll
  for (int p = 0; p < kChunks; p += 2) {
    chunk(ra, rb, p);
    chunk(rb, ra, p + 1);
  }
  return (m01.x + m01.y) + (m23.x + m23.y);
}

__device__ __forceinline__ void setup_sync(Sync& sy, int warp) {
  if (threadIdx.x == 0) {
    for (int s = 0; s < kP2Stages; ++s) {
      tc::mbar_init(&sy.a_full[s], 1);
      tc::mbar_init(&sy.a_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&sy.b_full[s], 1);
      tc::mbar_init(&sy.b_empty[s], 1);
      tc::mbar_init(&sy.acc_full[s], 1);
      tc::mbar_init(&sy.acc_empty[s], kEpiWarps);
    }
    tc::mbar_init(&sy.drain, 1);
    sy.abort = 0;
    tc::fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tc::tmem_alloc(&sy.tmem, kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
}

__device__ __forceinline__ void teardown(Sync& sy, int warp, uint32_t tmem, DevStatus* st) {
  tc::fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && sy.abort) record_error(st, AVTP_ERR_TIMEOUT, static_cast<int32_t>(blockIdx.x));
}

// ---------------------------------------------------------------- pass 1: log-sum-exp of every row
// mapQ: Qt {d, rows, Hkv}, box 64 x 128 x 1; mapK: keys {d, Hkv, T}, box 64 x 1 x 256.
__global__ void __launch_bounds__(kThreads, 1)
k_attn_lse(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK, AttnArgs a) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ Sync sy;
  __shared__ float2 s_mrg[2][2][kM];  // [segment parity][A tile][row]: column half 1's (max, sum)
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int d = a.d;
  unsigned char* sA = smem;  // A tile t at sA + t * a_bytes(d)
  unsigned char* sB[2] = {smem + 2 * a_bytes(d), smem + 2 * a_bytes(d) + b_bytes(d)};
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t atomA = kM * 128, atomB = kN * 128;  // bytes per 64-element atom column

  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int NB = a.blk_cu[a.R];
  const int F1 = a.meta[0], C1 = a.meta[1];
  const int64_t total = static_cast<int64_t>(a.Hkv) * F1;
  const int64_t f_begin = static_cast<int64_t>(blockIdx.x) * C1;
  if (f_begin >= total) return;
  const int n_steps = static_cast<int>(min(f_begin + C1, total) - f_begin);

  setup_sync(sy, warp);
  const uint32_t tmem = sy.tmem;
  volatile int* abort_flag = &sy.abort;
  FlatCursor cur;
  cur.init(f_begin, F1, a.p1s_cu, NB);

  if (warp == kTmaWarp) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tc::tma_prefetch_map(&mapQ);
      tc::tma_prefetch_map(&mapK);
      uint32_t na = 0, nb = 0;  // A (block) loads and B (key tile) loads issued so far
      int key_base = 0;
      bool new_seg = true;
      for (int st = 0; st < n_steps && !*abort_flag; ++st) {
        if (new_seg) {
          if (na >= 1 && !tc::mbar_wait(&sy.a_empty[0], (na - 1) & 1)) { *abort_flag = 1; break; }
          const Seg s = seg_of(a, cur.g, cur.b);
          tc::mbar_arrive_expect_tx(&sy.a_full[0], static_cast<uint32_t>(2 * a_bytes(d)));
          for (int t = 0; t < 2; ++t)
            for (int ac = 0; ac < d / 64; ++ac)
              tc::tma_load_3d(sA + t * a_bytes(d) + ac * atomA, &mapQ, ac * 64, static_cast<int>(s.R0) + t * kM,
                              cur.g, &sy.a_full[0]);
          ++na;
          key_base = a.cu[s.r];
        }
        const int sb = nb & 1;
        if (nb >= 2 && !tc::mbar_wait(&sy.b_empty[sb], ((nb >> 1) - 1) & 1)) { *abort_flag = 1; break; }
        tc::mbar_arrive_expect_tx(&sy.b_full[sb], static_cast<uint32_t>(b_bytes(d)));
        for (int ac = 0; ac < d / 64; ++ac)
          tc::tma_load_3d(sB[sb] + ac * atomB, &mapK, ac * 64, cur.g, key_base + cur.j * kN, &sy.b_full[sb]);
        attn_stamp(0, st, 0);
        ++nb;
        new_seg = st + 1 < n_steps && cur.next(a.p1s_cu, NB);
      }
      // let the copies in flight land before the CTA may exit
      if (na >= 1) tc::mbar_wait(&sy.a_full[0], (na - 1) & 1);
      for (uint32_t k = (nb >= 2 ? nb - 2 : 0); k < nb; ++k) tc::mbar_wait(&sy.b_full[k & 1], (k >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(kM, kN);
      uint32_t na = 0, nb = 0;
      bool new_seg = true, stop = false;
      for (int st = 0; st < n_steps && !stop && !*abort_flag; ++st) {
        attn_stamp(0, st, 1);
        if (new_seg) {
          if (!tc::mbar_wait(&sy.a_full[0], na & 1)) { *abort_flag = 1; break; }
          ++na;
        }
        const int sb = nb & 1;
        if (!tc::mbar_wait(&sy.b_full[sb], (nb >> 1) & 1)) { *abort_flag = 1; break; }
        for (int t = 0; t < 2; ++t) {
          // accumulator t: its previous use (step nb - 1) must have been read out
          if (nb >= 1 && !tc::mbar_wait(&sy.acc_empty[t], (nb - 1) & 1)) { *abort_flag = 1; stop = true; break; }
          if (t == 0) attn_stamp(0, st, 2);
          tc::fence_after_sync();
          tc::mma_rows(tmem + t * kN, tc::smem_u32(sA + t * a_bytes(d)), atomA, tc::smem_u32(sB[sb]), atomB, d, idesc);
          tc::mma_commit(&sy.acc_full[t]);
        }
        if (stop) break;
        tc::mma_commit(&sy.b_empty[sb]);
        attn_stamp(0, st, 3);
        ++nb;
        const bool more = st + 1 < n_steps;
        if (!more || cur.last_of_block()) tc::mma_commit(&sy.a_empty[0]);
        new_seg = more && cur.next(a.p1s_cu, NB);
      }
      // every MMA issued has completed once this arrives
      tc::mma_commit(&sy.drain);
      tc::mbar_wait(&sy.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue (8 warps)
    // Warp w reads TMEM lanes 32(w%4)..+31 (its rows of both A tiles) and columns
    // 128(w/4)..+127 of both accumulators; the two column halves of a row meet in
    // shared memory when the row's partial is written.
    const int quad = warp & 3, half = warp >> 2;
    const int lrow = quad * 32 + lane;  // row of each A tile = TMEM lane
    const uint32_t tbase = tmem + (static_cast<uint32_t>(quad * 32) << 16) + half * (kN / 2);
    const float c2 = a.c2;
    // After a timeout (abort_flag) the epilogue keeps walking the same steps, skipping
    // every wait and TMEM read, so that its named barriers still line up.
    int key_base = 0, qpos0 = -1, qpos1 = -1, par = 0;
    bool new_seg = true;
    float2* dst0 = nullptr;          // this row's partial (A tile 0, 1) of the current block
    float2* dst1 = nullptr;
    float m0 = -INFINITY, l0 = 0.f, m1 = -INFINITY, l1 = 0.f;  // running max and sum, log2 domain
    for (int st = 0; st < n_steps; ++st) {
      if (new_seg) {
        const Seg s = seg_of(a, cur.g, cur.b);
        key_base = a.cu[s.r];
        const int64_t F0 = static_cast<int64_t>(cur.g) * F1 + a.p1s_cu[cur.b];
        const int slot = static_cast<int>(blockIdx.x - F0 / C1);
        const int64_t row0 = s.R0 + lrow, row1 = s.R0 + kM + lrow;
        float2* base = a.p1_part + (static_cast<int64_t>(cur.g * NB + cur.b) * kBlk + lrow) * kAttnMaxChunks + slot;
        qpos0 = row0 < s.R1 ? a.text_idx[row0 / a.G] : -1;
        qpos1 = row1 < s.R1 ? a.text_idx[row1 / a.G] : -1;
        dst0 = row0 < s.R1 ? base : nullptr;
        dst1 = row1 < s.R1 ? base + static_cast<int64_t>(kM) * kAttnMaxChunks : nullptr;
        m0 = m1 = -INFINITY;
        l0 = l1 = 0.f;
      }
#pragma unroll 1
      for (int t = 0; t < 2; ++t) {
        bool ok = !__any_sync(0xffffffffu, *abort_flag != 0);
        if (ok && !tc::mbar_wait_warp(&sy.acc_full[t], st & 1)) {
          if (lane == 0) *abort_flag = 1;
          ok = false;
        }
        if (t == 0 && warp == 0 && lane == 0) attn_stamp(0, st, 4);
        tc::fence_after_sync();
        // columns 0..lim of this warp's half are visible to the row
        const int lim = (t ? qpos1 : qpos0) - (key_base + cur.j * kN + half * (kN / 2));
        const int lim_max = __reduce_max_sync(0xffffffffu, lim);
        if (ok && lim_max >= 0) {
          const uint32_t taddr = tbase + t * kN;
          float mt = t ? m1 : m0, lt = t ? l1 : l0;
          if (__all_sync(0xffffffffu, lim >= kHalf - 1)) {
            p1_slice<false>(taddr, kChunks, lim, c2, mt, lt);
          } else {
            // 32-column chunks 0 .. pe-1 hold a visible column for some lane
            p1_slice<true>(taddr, min(kChunks, (lim_max >> 5) + 1), lim, c2, mt, lt);
          }
          if (t) { m1 = mt; l1 = lt; } else { m0 = mt; l0 = lt; }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sy.acc_empty[t]);
        if (t == 1 && warp == 0 && lane == 0) attn_stamp(0, st, 5);
      }
      const bool more = st + 1 < n_steps;
      if (!more || cur.last_of_block()) {
        // the block ends here for this CTA: merge the column halves and write the partial
        par ^= 1;
        if (half == 1) {
          s_mrg[par][0][lrow] = make_float2(m0, l0);
          s_mrg[par][1][lrow] = make_float2(m1, l1);
        }
        bar_epi();
        if (half == 0) {
          auto merge = [&](float m, float l, float2 o, float2* dst) {
            const float M = fmaxf(m, o.x);
            const float L = (M == -INFINITY) ? 0.f : l * tc::ex2(m - M) + o.y * tc::ex2(o.x - M);
            *dst = make_float2(M, L);
          };
          if (dst0 != nullptr) merge(m0, l0, s_mrg[par][0][lrow], dst0);
          if (dst1 != nullptr) merge(m1, l1, s_mrg[par][1][lrow], dst1);
        }
      }
      new_seg = more && cur.next(a.p1s_cu, NB);
    }
  }
  teardown(sy, warp, tmem, a.st);
}

// ---------------------------------------------------------------- pass 2: probability mass of every visual key
// mapK: keys {d, Hkv, T}, box 64 x 1 x 128; mapQ: Qt {d, rows, Hkv}, box 64 x 256 x 1.
__global__ void __launch_bounds__(kThreads, 1)
k_attn_mass(const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapQ, AttnArgs a) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ Sync sy;
  __shared__ __align__(16) float s_lse[2][kBlk];  // -lse2, [block parity][row of the block]
  // key masses of the last steps, per column half, flushed to the accumulator every
  // kMassWindow steps (global atomics inside the step loop would be waited for by the
  // next step's TMEM fence)
  __shared__ float s_mass[kMassWindow][2][kM];
  __shared__ int s_tile[kMassWindow], s_nk[kMassWindow];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int d = a.d;
  unsigned char* sB = smem;  // the block's rows
  unsigned char* sA0 = smem + b_bytes(d);  // key tile s at sA0 + s * a_bytes(d)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t atomA = kM * 128, atomB = kN * 128;

  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int NB = a.blk_cu[a.R];
  const int F1 = a.meta[0], C1 = a.meta[1], F2 = a.meta[2], C2 = a.meta[3];
  const int64_t total = static_cast<int64_t>(a.Hkv) * F2;
  const int64_t f_begin = static_cast<int64_t>(blockIdx.x) * C2;
  if (f_begin >= total) return;
  const int n_steps = static_cast<int>(min(f_begin + C2, total) - f_begin);

  setup_sync(sy, warp);
  const uint32_t tmem = sy.tmem;
  volatile int* abort_flag = &sy.abort;
  FlatCursor cur;
  cur.init(f_begin, F2, a.p2t_cu, NB);

  if (warp == kTmaWarp) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tc::tma_prefetch_map(&mapQ);
      tc::tma_prefetch_map(&mapK);
      uint32_t na = 0, nbl = 0;  // key tile loads and block loads issued so far
      bool new_seg = true;
      Seg s{};
      TileCursor tile{};
      for (int st = 0; st < n_steps && !*abort_flag; ++st) {
        if (new_seg) {
          if (nbl >= 1 && !tc::mbar_wait(&sy.b_empty[0], (nbl - 1) & 1)) { *abort_flag = 1; break; }
          s = seg_of(a, cur.g, cur.b);
          tc::mbar_arrive_expect_tx(&sy.b_full[0], static_cast<uint32_t>(b_bytes(d)));
          for (int ac = 0; ac < d / 64; ++ac)
            tc::tma_load_3d(sB + ac * atomB, &mapQ, ac * 64, static_cast<int>(s.R0), cur.g, &sy.b_full[0]);
          ++nbl;
          tile.init(a, s, cur.j);
        } else {
          tile.next(a, s);
        }
        const int sa = na % kP2Stages;
        if (na >= kP2Stages && !tc::mbar_wait(&sy.a_empty[sa], ((na / kP2Stages) - 1) & 1)) { *abort_flag = 1; break; }
        tc::mbar_arrive_expect_tx(&sy.a_full[sa], static_cast<uint32_t>(a_bytes(d)));
        for (int ac = 0; ac < d / 64; ++ac)
          tc::tma_load_3d(sA0 + sa * a_bytes(d) + ac * atomA, &mapK, ac * 64, cur.g, tile.kp0, &sy.a_full[sa]);
        attn_stamp(1, st, 0);
        ++na;
        new_seg = st + 1 < n_steps && cur.next(a.p2t_cu, NB);
      }
      if (nbl >= 1) tc::mbar_wait(&sy.b_full[0], (nbl - 1) & 1);
      for (uint32_t k = (na >= kP2Stages ? na - kP2Stages : 0); k < na; ++k)
        tc::mbar_wait(&sy.a_full[k % kP2Stages], (k / kP2Stages) & 1);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(kM, kN);
      uint32_t na = 0, nbl = 0;
      bool new_seg = true;
      for (int st = 0; st < n_steps && !*abort_flag; ++st) {
        attn_stamp(1, st, 1);
        if (new_seg) {
          if (!tc::mbar_wait(&sy.b_full[0], nbl & 1)) { *abort_flag = 1; break; }
          ++nbl;
        }
        const int sa = na % kP2Stages;
        if (!tc::mbar_wait(&sy.a_full[sa], (na / kP2Stages) & 1)) { *abort_flag = 1; break; }
        const int t = na & 1;  // accumulator of this step
        if (na >= 2 && !tc::mbar_wait(&sy.acc_empty[t], ((na >> 1) - 1) & 1)) { *abort_flag = 1; break; }
        attn_stamp(1, st, 2);
        tc::fence_after_sync();
        tc::mma_rows(tmem + t * kN, tc::smem_u32(sA0 + sa * a_bytes(d)), atomA, tc::smem_u32(sB), atomB, d, idesc);
        tc::mma_commit(&sy.a_empty[sa]);
        tc::mma_commit(&sy.acc_full[t]);
        attn_stamp(1, st, 3);
        ++na;
        const bool more = st + 1 < n_steps;
        if (!more || cur.last_of_block()) tc::mma_commit(&sy.b_empty[0]);
        new_seg = more && cur.next(a.p2t_cu, NB);
      }
      tc::mma_commit(&sy.drain);
      tc::mbar_wait(&sy.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue (8 warps)
    // Warp w reads TMEM lanes 32(w%4)..+31 (its keys) and columns 128(w/4)..+127 (rows
    // of the block) of the step's accumulator; each column half adds its own share of a
    // key's mass to the fixed-point accumulator.
    const int quad = warp & 3, half = warp >> 2;
    const int klane = quad * 32 + lane;  // key of the tile = TMEM lane
    const int etid = threadIdx.x;        // 0 .. 255
    const uint32_t tbase = tmem + (static_cast<uint32_t>(quad * 32) << 16) + half * (kBlk / 2);
    const float c2 = a.c2;
    int par = 0, c1 = 0, img = -1;
    float lse_own = INFINITY;  // lse2 of this thread's row of the block (row etid)
    bool new_seg = true;
    Seg s{};
    TileCursor tile{};
    for (int st = 0; st < n_steps; ++st) {
      if (new_seg) {
        s = seg_of(a, cur.g, cur.b);
        c1 = static_cast<int>(s.R1 - s.R0);  // rows of the block that belong to the request
        const int g = cur.g, b = cur.b;
        const int64_t row = s.R0 + etid;
        lse_own = INFINITY;
        if (row < s.R1) {
          if (a.lse_rows != nullptr) {
            lse_own = a.lse_rows[static_cast<int64_t>(g) * a.rows + row];
          } else {
            // merge the row's pass-1 partials, eight loads in flight at a time
            const int64_t F0 = static_cast<int64_t>(g) * F1 + a.p1s_cu[b];
            const int steps = a.p1s_cu[b + 1] - a.p1s_cu[b];
            const int n = static_cast<int>((F0 + steps - 1) / C1 - F0 / C1) + 1;
            const float2* src = a.p1_part + (static_cast<int64_t>(g * NB + b) * kBlk + etid) * kAttnMaxChunks;
            float M = -INFINITY, L = 0.f;
            for (int k0 = 0; k0 < n; k0 += 8) {
              float2 pk[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) pk[k] = (k0 + k < n) ? src[k0 + k] : make_float2(-INFINITY, 0.f);
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const float Mn = fmaxf(M, pk[k].x);
                if (Mn != -INFINITY) {
                  L = L * tc::ex2(M - Mn) + pk[k].y * tc::ex2(pk[k].x - Mn);
                  M = Mn;
                }
              }
            }
            lse_own = M + __log2f(L);
          }
        }
        tile.init(a, s, cur.j);
        img = -1;
      } else {
        tile.next(a, s);
      }
      if (tile.i != img) {
        // the -lse2 vector of this (block, image): -inf on rows whose query precedes the
        // image, so that their terms vanish; double-buffered by parity
        img = tile.i;
        par ^= 1;
        s_lse[par][etid] = (etid >= tile.c0) ? -lse_own : -INFINITY;
        bar_epi();
      }
      const int t = st & 1;                                  // accumulator of this step
      const uint32_t use = static_cast<uint32_t>(st) >> 1;  // its use count
      bool ok = !__any_sync(0xffffffffu, *abort_flag != 0);
      if (ok && !tc::mbar_wait_warp(&sy.acc_full[t], use & 1)) {
        if (lane == 0) *abort_flag = 1;
        ok = false;
      }
      if (warp == 0 && lane == 0) attn_stamp(1, st, 4);
      tc::fence_after_sync();
      // does this warp's column half hold a visible row? (CTA-uniform)
      const bool any = tile.c0 < (half + 1) * kHalf && c1 > half * kHalf;
      float mass = 0.f;
      if (ok && any) mass = p2_slice(tbase + t * kN, &s_lse[par][half * kHalf], c2);
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sy.acc_empty[t]);
      if (warp == 0 && lane == 0) attn_stamp(1, st, 5);
      const int w = st % kMassWindow;
      s_mass[w][half][klane] = mass;
      if (etid == 0) {
        s_tile[w] = tile.tile;
        s_nk[w] = tile.nk;
      }
      if (w == kMassWindow - 1 || st + 1 == n_steps) {
        // flush: one fixed-point integer add per (step, key), both column halves summed
        // in fp32 first (integer adds: the result does not depend on their order)
        bar_epi();
        for (int e = etid; e < (w + 1) * kM; e += kEpiWarps * 32) {
          const int ws = e / kM, k = e % kM;
          if (k < s_nk[ws]) {
            const float m = s_mass[ws][0][k] + s_mass[ws][1][k];
            unsigned long long* dst = a.mass + static_cast<int64_t>(s_tile[ws]) * kM + k;
            if (m <= 512.f) {  // at most one per row of the block
              atomicAdd(dst, static_cast<unsigned long long>(__float2ll_rn(m * static_cast<float>(1ull << kAttnMassFracBits))));
            } else {
              atomicOr(dst, kMassNotFinite);  // NaN or inf inputs: the key scores NaN (bit 63; finite adds never reach it)
            }
          }
        }
        bar_epi();
      }
      new_seg = st + 1 < n_steps && cur.next(a.p2t_cu, NB);
    }
  }
  teardown(sy, warp, tmem, a.st);
}

// ---------------------------------------------------------------- repacking of the text queries
// Qt[g][o*G + j][:] = q[text_idx[o], g*G + j, :]; with a supplied LSE also
// lse_rows[g][o*G + j] = lse[g*G + j][text_idx[o]] * log2(e). One thread per 16 bytes.
// Also clears the per-key mass accumulator of pass 2.
__global__ void __launch_bounds__(256)
k_attn_pack(const __nv_bfloat16* __restrict__ q, int64_t q_stride, int Hq, int G, int d,
            const int32_t* __restrict__ text_idx, const int32_t* __restrict__ text_cu, int R, int64_t rows,
            __nv_bfloat16* __restrict__ qt, const float* __restrict__ lse, int64_t lse_stride,
            float* __restrict__ lse_rows, unsigned long long* __restrict__ mass, int64_t n_mass, const DevStatus* st) {
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int64_t n_text = text_cu[R];
  const int vec = d / 8;
  const int64_t total = n_text * Hq * vec;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t tid0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  for (int64_t u = tid0; u < n_mass; u += stride) mass[u] = 0ull;
  for (int64_t u = tid0; u < total; u += stride) {
    const int c = static_cast<int>(u % vec);
    const int64_t oh = u / vec;
    const int h = static_cast<int>(oh % Hq);
    const int64_t o = oh / Hq;
    const int g = h / G, j = h - g * G;
    const int64_t pos = text_idx[o];
    const int64_t row = o * G + j;
    const uint4 v = *reinterpret_cast<const uint4*>(q + pos * q_stride + static_cast<int64_t>(h) * d + c * 8);
    *reinterpret_cast<uint4*>(qt + (static_cast<int64_t>(g) * rows + row) * d + c * 8) = v;
    if (lse != nullptr && c == 0) lse_rows[static_cast<int64_t>(g) * rows + row] = lse[h * lse_stride + pos] * kLog2e;
  }
}

// ---------------------------------------------------------------- finalize
// One CTA per key tile (128 keys of one image): s_t = mass_t * 2^-40 / (Hq * |Q_r|), and
// the tile's fixed-point score sum added to its image's sum with one atomic.
__global__ void __launch_bounds__(kM)
k_attn_finalize(const unsigned long long* __restrict__ mass, const int32_t* __restrict__ ktile_cu,
                const int32_t* __restrict__ ktile_img, int Hq, const int32_t* __restrict__ cu,
                const int32_t* __restrict__ img_start, const int32_t* __restrict__ img_len,
                const int32_t* __restrict__ img_req, const int32_t* __restrict__ text_cu, int NI, int last,
                float* __restrict__ scores, int64_t* __restrict__ img_sums, const DevStatus* st) {
  __shared__ long long s_part[kM / 32];
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  for (int tile = blockIdx.x; tile < ktile_cu[NI]; tile += gridDim.x) {
    const int i = ktile_img[tile];
    const int r = img_req[i];
    const int o = (tile - ktile_cu[i]) * kM + static_cast<int>(threadIdx.x);  // key within the image
    // the request's queries: its text tokens, or its last token alone
    const int nq = last ? (cu[r + 1] > cu[r] ? 1 : 0) : text_cu[r + 1] - text_cu[r];
    const unsigned long long m = mass[static_cast<int64_t>(tile) * kM + threadIdx.x];
    long long fx = 0;
    if (o < img_len[i]) {
      float s = 0.f;
      if (nq > 0) {
        if (m & kMassNotFinite) {
          s = __int_as_float(0x7fc00000);
        } else {
          s = __ll2float_rn(static_cast<long long>(m)) * (1.0f / static_cast<float>(1ull << kAttnMassFracBits));
          s = s / static_cast<float>(static_cast<int64_t>(Hq) * nq);
        }
      }
      scores[static_cast<int64_t>(cu[r]) + img_start[i] + o] = s;
      fx = fixed_point_score(s);
    }
    fx = warp_sum(fx);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = fx;
    __syncthreads();
    if (threadIdx.x == 0) {
      long long sum = 0;
#pragma unroll
      for (int w = 0; w < kM / 32; ++w) sum += s_part[w];
      atomicAdd(reinterpret_cast<unsigned long long*>(img_sums + i), static_cast<unsigned long long>(sum));
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

// A 3-D bf16 tensor map with 128-byte swizzle and a box of 64 x box1 x box2 elements.
bool make_map(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t stride1_bytes,
              uint64_t stride2_bytes, uint32_t box1, uint32_t box2) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {64, box1, box2};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_score_attn(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                              int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s) {
  if (L.n_images == 0 || L.n_tokens == 0) return cudaSuccess;
  const int d = sa.head_dim, Hq = sa.n_q_heads, Hkv = sa.n_kv_heads;
  const AttnPlan plan = attn_plan(L, sa);
  static PerDevice attrs;
  cudaError_t ae = once_per_device(attrs, [](int, int*) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_lse, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(lse_smem_bytes(128)));
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_attn_mass, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(mass_smem_bytes(128)));
  });
  if (ae != cudaSuccess) return ae;
  DevStatus* st = ws_at<DevStatus>(ws, p.status);
  AttnArgs a{};
  a.cu = L.cu_seqlens;
  a.R = L.n_requests;
  a.ist = L.img_start;
  a.iln = L.img_len;
  a.icu = L.img_cu;
  a.NI = L.n_images;
  a.T = L.n_tokens;
  a.vis_cu = ws_at<int32_t>(ws, p.vis_cu);
  a.text_idx = ws_at<int32_t>(ws, p.text_idx);
  a.text_cu = ws_at<int32_t>(ws, p.text_cu);
  a.blk_cu = ws_at<int32_t>(ws, p.blk_cu);
  a.p1s_cu = ws_at<int32_t>(ws, p.p1s_cu);
  a.p2t_cu = ws_at<int32_t>(ws, p.p2t_cu);
  a.ktile_cu = ws_at<int32_t>(ws, p.ktile_cu);
  a.meta = ws_at<int32_t>(ws, p.meta);
  float* lse_rows = sa.lse != nullptr ? ws_at<float>(ws, p.lse_rows) : nullptr;
  a.lse_rows = lse_rows;
  a.p1_part = sa.lse == nullptr ? ws_at<float2>(ws, p.p1_part) : nullptr;
  a.mass = ws_at<unsigned long long>(ws, p.mass);
  a.rows = plan.rows;
  a.G = plan.G;
  a.Hkv = Hkv;
  a.d = d;
  a.c2 = sa.softmax_scale * kLog2e;
  a.st = st;
  __nv_bfloat16* qt = ws_at<__nv_bfloat16>(ws, p.qt);

  // tensor maps: keys {d, Hkv, T} (token stride k_stride), packed queries {d, rows, Hkv}
  CUtensorMap mk128, mk256, mq128, mq256;
  const uint64_t ks = static_cast<uint64_t>(sa.k_stride) * 2, qs = static_cast<uint64_t>(plan.rows) * d * 2;
  if (!make_map(&mk128, sa.k, d, Hkv, L.n_tokens, static_cast<uint64_t>(d) * 2, ks, 1, kM) ||
      !make_map(&mk256, sa.k, d, Hkv, L.n_tokens, static_cast<uint64_t>(d) * 2, ks, 1, kN) ||
      !make_map(&mq128, qt, d, plan.rows, Hkv, static_cast<uint64_t>(d) * 2, qs, kM, 1) ||
      !make_map(&mq256, qt, d, plan.rows, Hkv, static_cast<uint64_t>(d) * 2, qs, kBlk, 1))
    return cudaErrorInvalidValue;

  const int sms = plan.grid;
  {
    const int64_t want = (plan.max_text * Hq * (d / 8) + 255) / 256;
    const int64_t cap = static_cast<int64_t>(sms) * 8;
    const int grid = static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
    cudaError_t e = launch_kernel(k_attn_pack, dim3(grid), dim3(256), 0, s, /*pdl=*/true,
                                  static_cast<const __nv_bfloat16*>(sa.q), sa.q_stride, Hq, plan.G, d, a.text_idx,
                                  a.text_cu, L.n_requests, plan.rows, qt, sa.lse, sa.lse_stride, lse_rows, a.mass,
                                  plan.n_ktiles_max * kM, static_cast<const DevStatus*>(st));
    if (e != cudaSuccess) return e;
  }
  if (sa.lse == nullptr) {
    cudaError_t e = launch_kernel(k_attn_lse, dim3(sms), dim3(kThreads), lse_smem_bytes(d), s, /*pdl=*/true, mq128,
                                  mk256, a);
    if (e != cudaSuccess) return e;
  }
  cudaError_t e =
      launch_kernel(k_attn_mass, dim3(sms), dim3(kThreads), mass_smem_bytes(d), s, /*pdl=*/true, mk128, mq256, a);
  if (e != cudaSuccess) return e;
  return launch_attn_finalize(L, sa, scores, img_sums, ws, p, plan, s);
}

cudaError_t launch_attn_finalize(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                                 int64_t* img_sums, void* ws, const WsPlan& p, const AttnPlan& plan, cudaStream_t s) {
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  const int grid3 = static_cast<int>(plan.n_ktiles_max < cap ? plan.n_ktiles_max : cap);
  return launch_kernel(k_attn_finalize, dim3(grid3), dim3(kM), 0, s, /*pdl=*/true,
                       static_cast<const unsigned long long*>(ws_at<unsigned long long>(ws, p.mass)),
                       static_cast<const int32_t*>(ws_at<int32_t>(ws, p.ktile_cu)),
                       static_cast<const int32_t*>(ws_at<int32_t>(ws, p.ktile_img)), sa.n_q_heads, L.cu_seqlens,
                       L.img_start, L.img_len, static_cast<const int32_t*>(ws_at<int32_t>(ws, p.img_req)),
                       static_cast<const int32_t*>(ws_at<int32_t>(ws, p.text_cu)), L.n_images,
                       sa.query_set == AVTP_QUERIES_LAST ? 1 : 0, scores, img_sums,
                       static_cast<const DevStatus*>(ws_at<DevStatus>(ws, p.status)));
}

}  // namespace avtp

extern "C" avtp_status_t avtp_score_timeline(int32_t pass, int64_t* out, int32_t max_steps) {
#ifdef AVTP_TIMELINE
  if (out == nullptr || max_steps < 1 || (pass != 1 && pass != 2)) return AVTP_ERR_INVALID_ARG;
  const int n = max_steps < avtp::kAttnTlSteps ? max_steps : avtp::kAttnTlSteps;
  const size_t row = static_cast<size_t>(avtp::kAttnTlSteps) * avtp::kAttnTlSlots * sizeof(long long);
  return cudaMemcpyFromSymbol(out, avtp::g_attn_tl, static_cast<size_t>(n) * avtp::kAttnTlSlots * sizeof(long long),
                              (pass - 1) * row) == cudaSuccess
             ? AVTP_OK
             : AVTP_ERR_CUDA;
#else
  (void)pass;
  (void)out;
  (void)max_steps;
  return AVTP_ERR_UNSUPPORTED;
#endif
}
