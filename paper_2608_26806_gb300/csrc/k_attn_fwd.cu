// The pruning layer's causal attention forward (paper §3.2: the FlashAttention-style
// forward whose natural-log normaliser the text-attention criterion reuses), on a
// varlen-packed batch with grouped-query heads g(h) = h / (Hq / Hkv), head_dim 64 or 128:
//   O[t, h]   = sum_{u visible to t} softmax_u(scale * q[t, h] . k[u, g(h)]) v[u, g(h)]
//   lse[h, t] = ln sum_{u visible to t} exp(scale * q[t, h] . k[u, g(h)])
// where u is visible to t when it lies in t's request and u <= t.
//
// A CTA owns one tile of 128 query tokens of one request and one query head. Its key
// blocks of 128 keys are aligned to multiples of 128 in the packed token index (so that
// every TMA x coordinate into the transposed values is a multiple of 64), from the block
// of the request's first token to the block of the tile's last token; keys outside the
// request or after the query are masked.
//
// Per key block j:
//   S_j = Q K_j^T           tcgen05 with A (Q) read from TMEM, M = 128 queries, N = 128 keys
//   P_j = exp2(c2 S_j - m)  softmax warps; bf16, two per column, into a TMEM P buffer
//   O  += P_j V_j           tcgen05 with A (P) read from TMEM, M = 128, N = d, K = 128 keys
// with c2 = scale * log2(e). A row's reference max m moves only when a block's max
// exceeds it by more than 8 (log2 units), so the accumulator in TMEM is rescaled rarely
// and every P entry stays below 2^8. P V needs V with keys contiguous (the MMA's K-major
// operand), so a first kernel writes the values transposed, Vt[g][c][t].
//
// Warps 0-7: softmax and epilogue. Warp w owns query rows 32 (w % 4) .. + 31 (TMEM lanes)
// and key half w / 4 of every block, so two warps share every SM sub-partition; the two
// warps of a row range exchange their half maxima through shared memory once per block
// (a 64-thread named barrier), so a row has one reference max and one accumulator. Warp
// 8 issues the TMA loads (Q once, K and Vt double-buffered). Warp 9 owns TMEM and issues
// the MMAs in the order S_{j+1}, P_j V_j: S_{j+1} as soon as the softmax has read S_j
// out of TMEM, P_j V_j once P_j is written, so the tensor core has the next block's work
// queued while the softmax runs. One thread issues every MMA, and an MMA is issued no
// faster than the tensor core takes its operands, so the operands come from TMEM where
// they can: Q (copied there once by the softmax warps) and P are the A operands, and
// only K and V are read from shared memory. TMEM: S in columns 0-127, P buffers in
// 128-255 (64 columns each), Q in 256-319, O in 384 .. 384 + d.
// Every wait is bounded; a CTA whose wait gives up records AVTP_ERR_TIMEOUT and returns.
#include <cudaTypedefs.h>

#include "avtp_fwd.cuh"
#include "avtp_tc.cuh"

namespace avtp {
namespace {

constexpr int kQT = 128;  // query rows per tile (MMA M, TMEM lanes)
constexpr int kKB = 128;  // keys per block (MMA N of Q K^T, K of P V)
constexpr int kHalf = kKB / 2;  // keys of a block per softmax warp
constexpr int kThreads = 320;
constexpr int kSoftWarps = 8;
constexpr int kTmaWarp = 8;
constexpr int kMmaWarp = 9;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSCol = 0;
constexpr uint32_t kPCol = 128;  // P buffer b at kPCol + 64 b (two bf16 per column)
constexpr uint32_t kQCol = 256;  // Q, two bf16 per column (d / 2 columns)
constexpr uint32_t kOCol = 384;
constexpr float kRescaleTau = 8.f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLog2e = 1.4426950408889634f;

__host__ __device__ constexpr size_t q_bytes(int d) { return static_cast<size_t>(kQT) * d * 2; }
__host__ __device__ constexpr size_t k_bytes(int d) { return static_cast<size_t>(kKB) * d * 2; }
__host__ __device__ constexpr size_t v_bytes(int d) { return static_cast<size_t>(d) * kKB * 2; }
__host__ __device__ constexpr size_t fwd_smem_bytes(int d) { return 1024 + q_bytes(d) + 2 * k_bytes(d) + 2 * v_bytes(d); }
// Every head_dim requests more than half the SM's shared memory, so that no second CTA
// (and its 512 TMEM columns) shares an SM.
constexpr size_t kFwdSmem = fwd_smem_bytes(128) > 116 * 1024 ? fwd_smem_bytes(128) : 116 * 1024;
static_assert(kFwdSmem <= 227 * 1024, "shared memory of one CTA");

struct FwdSync {
  uint64_t q_full;
  uint64_t k_full[2], k_empty[2];
  uint64_t v_full[2], v_empty[2];
  uint64_t q_tmem;                 // Q copied into TMEM by the softmax warps
  uint64_t s_full, s_empty;        // S: written by the MMA / read out by the softmax
  uint64_t p_full[2], pv_done[2];  // P buffer b: written by the softmax / read by P V
  uint64_t drain;
  uint32_t tmem;
  int abort;
};

struct FwdArgs {
  const int32_t* cu;
  int R;
  const int32_t* qtile_cu;
  int Hq, G, d;
  float c2;
  float* o;
  int64_t o_stride;
  float* lse;
  int64_t lse_stride;
  DevStatus* st;
};

// 32 consecutive fp32 columns of this thread's TMEM lane, stored; complete after
// tmem_wait_st().
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
      "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
      "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// D[tmem] (+)= A[tmem] * B^T for one K = 16 step, A (M x 16, two bf16 per column) read
// from tensor memory; issued by a single thread.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Diagnostic timeline build (-DAVTP_TIMELINE): clock stamps of the grid's first CTA (the
// tile with the most key blocks, head 0), per key block j. Slots: 0-4 from softmax warp 0
// (loop top, S ready, half maxima exchanged, exponentials done, P handed over); 5-9 from
// the MMA thread (S_j: entry, issued; P_j V_j: entry, operands ready, issued). Read with
// avtp_forward_timeline().
constexpr int kFwdTlBlocks = 256;
constexpr int kFwdTlSlots = 10;
#ifdef AVTP_TIMELINE
__device__ long long g_fwd_tl[kFwdTlBlocks][kFwdTlSlots];
#endif
__device__ __forceinline__ void fwd_stamp(int j, int slot) {
#ifdef AVTP_TIMELINE
  if (blockIdx.x == 0 && j < kFwdTlBlocks) g_fwd_tl[j][slot] = clock64();
#else
  (void)j;
  (void)slot;
#endif
}

__device__ __forceinline__ void bar_softmax() { asm volatile("bar.sync 5, 256;" ::: "memory"); }
// Barrier of the two softmax warps of TMEM lane quadrant `quad` (ids 1-4, 64 threads); true
// when `bad` holds for any of their threads.
__device__ __forceinline__ bool bar_pair_any(int quad, bool bad) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %2, 0;\n\t"
      "barrier.red.or.pred q, %1, 64, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(1 + quad), "r"(bad ? 1u : 0u)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&b);
}

// ---------------------------------------------------------------- forward
// mapQ: q {d, Hq, T}, box 64 x 1 x 128; mapK: k {d, Hkv, T}, box 64 x 1 x 128;
// mapV: Vt {Tp, d, Hkv}, box 64 x d x 1.
__global__ void __launch_bounds__(kThreads, 1)
k_attn_fwd(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
           const __grid_constant__ CUtensorMap mapV, FwdArgs a) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ FwdSync sy;
  __shared__ float2 s_ml[2][kQT];    // (reference max, sum over the half) of each row, at the end
  __shared__ float s_mx[2][2][kQT];   // [S buffer][key half][row]: block max of the half
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int d = a.d;
  unsigned char* sQ = smem;
  // key stage b at sK + b * k_bytes(d), value stage b at sV + b * v_bytes(d)
  unsigned char* sK = sQ + q_bytes(d);
  unsigned char* sV = sK + 2 * k_bytes(d);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int NQT = a.qtile_cu[a.R];
  const int u = static_cast<int>(blockIdx.x) / a.Hq;
  const int h = static_cast<int>(blockIdx.x) - u * a.Hq;
  if (u >= NQT) return;
  const int tq = NQT - 1 - u;  // the tiles with the most key blocks first
  const int r = upper_index(a.qtile_cu, a.R, tq);
  const int cu_r = a.cu[r];
  const int q0 = cu_r + (tq - a.qtile_cu[r]) * kQT;
  const int q_last = min(q0 + kQT, a.cu[r + 1]) - 1;
  const int kb0 = cu_r / kKB;
  const int nblk = q_last / kKB - kb0 + 1;
  const int g = h / a.G;

  if (threadIdx.x == 0) {
    tc::mbar_init(&sy.q_full, 1);
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&sy.k_full[s], 1);
      tc::mbar_init(&sy.k_empty[s], 1);
      tc::mbar_init(&sy.v_full[s], 1);
      tc::mbar_init(&sy.v_empty[s], 1);
      tc::mbar_init(&sy.p_full[s], kSoftWarps);
      tc::mbar_init(&sy.pv_done[s], 1);
    }
    tc::mbar_init(&sy.q_tmem, kSoftWarps);
    tc::mbar_init(&sy.s_full, 1);
    tc::mbar_init(&sy.s_empty, kSoftWarps);
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
  const uint32_t tmem = sy.tmem;
  volatile int* abort_flag = &sy.abort;

  if (warp == kTmaWarp) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tc::tma_prefetch_map(&mapQ);
      tc::tma_prefetch_map(&mapK);
      tc::tma_prefetch_map(&mapV);
      tc::mbar_arrive_expect_tx(&sy.q_full, static_cast<uint32_t>(q_bytes(d)));
      for (int ac = 0; ac < d / 64; ++ac) tc::tma_load_3d(sQ + ac * (kQT * 128), &mapQ, ac * 64, h, q0, &sy.q_full);
      int nk = 0, nv = 0;  // key and value blocks issued
      for (int j = 0; j < nblk && !*abort_flag; ++j) {
        const int sb = j & 1;
        const int key0 = (kb0 + j) * kKB;
        if (j >= 2 && !tc::mbar_wait(&sy.k_empty[sb], ((j >> 1) - 1) & 1)) { *abort_flag = 1; break; }
        tc::mbar_arrive_expect_tx(&sy.k_full[sb], static_cast<uint32_t>(k_bytes(d)));
        for (int ac = 0; ac < d / 64; ++ac)
          tc::tma_load_3d(sK + sb * k_bytes(d) + ac * (kKB * 128), &mapK, ac * 64, g, key0, &sy.k_full[sb]);
        ++nk;
        if (j >= 2 && !tc::mbar_wait(&sy.v_empty[sb], ((j >> 1) - 1) & 1)) { *abort_flag = 1; break; }
        tc::mbar_arrive_expect_tx(&sy.v_full[sb], static_cast<uint32_t>(v_bytes(d)));
        for (int kc = 0; kc < kKB / 64; ++kc)
          tc::tma_load_3d(sV + sb * v_bytes(d) + kc * (d * 128), &mapV, key0 + kc * 64, 0, g, &sy.v_full[sb]);
        ++nv;
      }
      // let the copies in flight land before the CTA may exit
      tc::mbar_wait(&sy.q_full, 0);
      for (int k = (nk >= 2 ? nk - 2 : 0); k < nk; ++k) tc::mbar_wait(&sy.k_full[k & 1], (k >> 1) & 1);
      for (int k = (nv >= 2 ? nv - 2 : 0); k < nv; ++k) tc::mbar_wait(&sy.v_full[k & 1], (k >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idS = tc::idesc_bf16(kQT, kKB), idO = tc::idesc_bf16(kQT, d);
      // S_j = Q K_j^T into S, once the softmax has read S_{j-1} out of it: A = Q in TMEM
      // (128 lanes x d / 2 columns), B = key stage j % 2 (128 keys x d, K-major)
      auto issue_s = [&](int j) -> bool {
        const int sb = j & 1;
        fwd_stamp(j, 5);
        if (!tc::mbar_wait(&sy.k_full[sb], (j >> 1) & 1)) return false;
        if (j >= 1 && !tc::mbar_wait(&sy.s_empty, (j - 1) & 1)) return false;
        tc::fence_after_sync();
        const uint32_t bK = tc::smem_u32(sK + sb * k_bytes(d));
        for (int ks = 0; ks < d / 16; ++ks) {
          const uint32_t bp = bK + static_cast<uint32_t>((ks >> 2) * (kKB * 128) + (ks & 3) * 32);
          mma_bf16_ts(tmem + kSCol, tmem + kQCol + static_cast<uint32_t>(ks * 8), tc::desc_k_sw128(bp), idS,
                      ks > 0 ? 1u : 0u);
        }
        tc::mma_commit(&sy.s_full);
        tc::mma_commit(&sy.k_empty[sb]);
        fwd_stamp(j, 6);
        return true;
      };
      // O += P_i V_i: A = P buffer i % 2 in TMEM (128 lanes x 64 columns), B = the Vt block
      // (d rows x 128 keys, two 64-key panels)
      auto issue_pv = [&](int i) -> bool {
        const int sb = i & 1;
        fwd_stamp(i, 7);
        if (!tc::mbar_wait(&sy.p_full[sb], (i >> 1) & 1)) return false;
        if (!tc::mbar_wait(&sy.v_full[sb], (i >> 1) & 1)) return false;
        fwd_stamp(i, 8);
        tc::fence_after_sync();
        const uint32_t bV = tc::smem_u32(sV + sb * v_bytes(d));
#pragma unroll
        for (int ks = 0; ks < kKB / 16; ++ks) {
          const uint32_t ap = tmem + kPCol + static_cast<uint32_t>(sb * 64 + ks * 8);
          const uint32_t bp = bV + static_cast<uint32_t>((ks >> 2) * (d * 128) + (ks & 3) * 32);
          mma_bf16_ts(tmem + kOCol, ap, tc::desc_k_sw128(bp), idO, (i > 0 || ks > 0) ? 1u : 0u);
        }
        tc::mma_commit(&sy.pv_done[sb]);
        tc::mma_commit(&sy.v_empty[sb]);
        fwd_stamp(i, 9);
        return true;
      };
      bool ok = tc::mbar_wait(&sy.q_tmem, 0) && issue_s(0);
      for (int j = 0; ok && j < nblk && !*abort_flag; ++j) {
        if (j + 1 < nblk && !issue_s(j + 1)) { ok = false; break; }
        if (!issue_pv(j)) { ok = false; break; }
      }
      if (!ok) *abort_flag = 1;
      // every MMA issued has completed once this arrives
      tc::mma_commit(&sy.drain);
      tc::mbar_wait(&sy.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ softmax and epilogue (warps 0-7)
    const int quad = warp & 3, half = warp >> 2;
    const int row = quad * 32 + lane;
    const int qpos = q0 + row;
    const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16);  // this warp's TMEM lanes
    const int oc0 = half * (d / 2);  // O columns this warp rescales and writes out
    const float c2 = a.c2;
    const float2 cc = make_float2(c2, c2);
    float m = -INFINITY, l = 0.f;  // row reference max (log2 units); sum of exp2(c2 s - m) over this half
    bool bad = false;               // a wait gave up (here or, through the pair barrier, in the partner)
    // Q into TMEM: warp (quad, half) copies 64-element panel `half` of its 32 rows (d = 64:
    // half 0 alone), unswizzling the 128-byte TMA layout (16-byte chunk c of row r at
    // chunk position c ^ (r % 8))
    if (!tc::mbar_wait_warp(&sy.q_full, 0)) bad = true;
    if (!bad && half < d / 64) {
      const unsigned char* qrow = sQ + half * (kQT * 128) + row * 128;
      uint32_t qv[32];
#pragma unroll
      for (int c16 = 0; c16 < 8; ++c16) {
        const uint4 u = *reinterpret_cast<const uint4*>(qrow + ((c16 ^ (row & 7)) << 4));
        qv[4 * c16] = u.x;
        qv[4 * c16 + 1] = u.y;
        qv[4 * c16 + 2] = u.z;
        qv[4 * c16 + 3] = u.w;
      }
      tmem_st32(tl + kQCol + half * 32, qv);
      tmem_wait_st();
    }
    tc::fence_before_sync();
    __syncwarp();
    if (!bad && lane == 0) tc::mbar_arrive(&sy.q_tmem);
    for (int j = 0; j < nblk; ++j) {
      const int sb = j & 1;
      const int key0 = (kb0 + j) * kKB + half * kHalf;
      const bool stamp = warp == 0 && lane == 0;
      if (stamp) fwd_stamp(j, 0);
      bad = bad || __any_sync(0xffffffffu, *abort_flag != 0);
      if (!bad && !tc::mbar_wait_warp(&sy.s_full, j & 1)) bad = true;
      if (stamp) fwd_stamp(j, 1);
      float s[kHalf];
      float mh = -INFINITY;
      if (!bad) {
        tc::fence_after_sync();
        tc::tmem_ld64(tl + kSCol + half * kHalf, s);
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sy.s_empty);
        // key key0 + c is visible to this row when cu_r <= key0 + c <= qpos
        const int lo = cu_r - key0, hi = qpos - key0;
        if (__any_sync(0xffffffffu, lo > 0 || hi < kHalf - 1)) {
#pragma unroll
          for (int c = 0; c < kHalf; ++c) s[c] = (c >= lo && c <= hi) ? s[c] : -INFINITY;
        }
        // max: eight running maxima (columns c mod 8), then their tree; exact in any order
        float t[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) t[c] = s[c];
#pragma unroll
        for (int c = 8; c < kHalf; ++c) t[c & 7] = fmaxf(t[c & 7], s[c]);
#pragma unroll
        for (int w = 4; w >= 1; w >>= 1) {
#pragma unroll
          for (int c = 0; c < w; ++c) t[c] = fmaxf(t[c], t[c + w]);
        }
        mh = t[0];
      }
      // the row's block max from both halves; both warps of the pair leave together
      s_mx[sb][half][row] = mh;
      if (bar_pair_any(quad, bad)) {
        if (lane == 0) *abort_flag = 1;
        break;
      }
      if (stamp) fwd_stamp(j, 2);
      const float mb = fmaxf(mh, s_mx[sb][half ^ 1][row]) * c2;  // -inf when nothing is visible
      float factor = 1.f;
      bool resc = false;
      if (mb > m + kRescaleTau) {
        if (m != -INFINITY) {
          factor = tc::ex2(m - mb);
          resc = true;
        }
        l *= factor;
        m = mb;
      }
      const float nm = (m == -INFINITY) ? 0.f : -m;
      const float2 nn = make_float2(nm, nm);
      uint32_t pk[kHalf / 2];
      float2 acc0 = make_float2(0.f, 0.f), acc1 = acc0;
#pragma unroll
      for (int c = 0; c < kHalf; c += 4) {
        const float2 z01 = tc::ffma2(make_float2(s[c], s[c + 1]), cc, nn);
        const float2 z23 = tc::ffma2(make_float2(s[c + 2], s[c + 3]), cc, nn);
        const float p0 = tc::ex2(z01.x), p1 = tc::ex2(z01.y), p2 = tc::ex2(z23.x), p3 = tc::ex2(z23.y);
        acc0 = tc::add2(acc0, make_float2(p0, p1));
        acc1 = tc::add2(acc1, make_float2(p2, p3));
        pk[c / 2] = pack_bf16x2(p0, p1);
        pk[c / 2 + 1] = pack_bf16x2(p2, p3);
      }
      l += (acc0.x + acc0.y) + (acc1.x + acc1.y);
      if (stamp) fwd_stamp(j, 3);
      // O is final up to block j - 1 once P_{j-1} V_{j-1} is done: a rescale waits for it and
      // scales this warp's half of the columns (both warps of the pair took the same factor)
      if (j >= 1 && __any_sync(0xffffffffu, resc)) {
        if (!tc::mbar_wait_warp(&sy.pv_done[(j - 1) & 1], ((j - 1) >> 1) & 1)) {
          bad = true;
          continue;  // to the next pair barrier, where both warps stop
        }
        tc::fence_after_sync();
        for (int oc = 0; oc < d / 64; ++oc) {
          uint32_t ov[32];
          tc::tmem_ld32_async(tl + kOCol + oc0 + oc * 32, ov);
          tc::tmem_wait(ov);
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * factor);
          tmem_st32(tl + kOCol + oc0 + oc * 32, ov);
        }
        tmem_wait_st();
      }
      // P buffer sb is free once P_{j-2} V_{j-2} has completed
      if (j >= 2 && !tc::mbar_wait_warp(&sy.pv_done[sb], ((j >> 1) - 1) & 1)) {
        bad = true;
        continue;
      }
      tc::fence_after_sync();
      tmem_st32(tl + kPCol + sb * 64 + half * 32, pk);
      tmem_wait_st();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sy.p_full[sb]);
      if (stamp) fwd_stamp(j, 4);
    }
    bool fin = !bad && !__any_sync(0xffffffffu, *abort_flag != 0);
    if (fin && !tc::mbar_wait_warp(&sy.pv_done[(nblk - 1) & 1], ((nblk - 1) >> 1) & 1)) {
      if (lane == 0) *abort_flag = 1;
      fin = false;
    }
    // the row's sum over both halves; every softmax warp passes this barrier once
    s_ml[half][row] = make_float2(m, l);
    bar_softmax();
    if (fin) {
      tc::fence_after_sync();
      const float L = s_ml[0][row].y + s_ml[1][row].y;
      const float inv = L > 0.f ? 1.f / L : 0.f;
      const bool live = qpos <= q_last;
      float* orow = a.o + static_cast<int64_t>(qpos) * a.o_stride + static_cast<int64_t>(h) * d + oc0;
      for (int oc = 0; oc < d / 64; ++oc) {
        float v[32];
        tc::tmem_ld32(tl + kOCol + oc0 + oc * 32, v);
        if (live) {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            *reinterpret_cast<float4*>(orow + oc * 32 + 4 * i) =
                make_float4(v[4 * i] * inv, v[4 * i + 1] * inv, v[4 * i + 2] * inv, v[4 * i + 3] * inv);
        }
      }
      if (live && half == 0) a.lse[static_cast<int64_t>(h) * a.lse_stride + qpos] = (m + log2f(L)) * kLn2;
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && sy.abort) record_error(a.st, AVTP_ERR_TIMEOUT, static_cast<int32_t>(blockIdx.x));
}

// ---------------------------------------------------------------- transposed values
// Vt[g][c][t] = v[t][g][c] for t < T and 0 for T <= t < Tp. A CTA moves a tile of 64
// tokens x 64 channels of one KV head through shared memory, 16 bytes per global access on
// both sides. The tile is read down its columns, so its 16-byte chunks are swizzled: chunk
// c of token row t sits at chunk position c ^ (t / 8 % 8), and the eight token rows a warp
// reads at once fall on different banks.
__global__ void __launch_bounds__(256)
k_attn_vt(const __nv_bfloat16* __restrict__ v, int64_t v_stride, int d, int64_t T, int64_t Tp,
          __nv_bfloat16* __restrict__ vt, const DevStatus* st) {
  __shared__ __align__(16) uint16_t tile[64][64];  // [token][channel], swizzled 16-byte chunks
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * 64;
  const int c0 = static_cast<int>(blockIdx.y) * 64;
  const int g = static_cast<int>(blockIdx.z);
  for (int e = threadIdx.x; e < 64 * 8; e += blockDim.x) {
    const int tt = e >> 3, ch = e & 7;
    const int64_t t = t0 + tt;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (t < T) val = *reinterpret_cast<const uint4*>(v + t * v_stride + static_cast<int64_t>(g) * d + c0 + ch * 8);
    *reinterpret_cast<uint4*>(&tile[tt][(ch ^ ((tt >> 3) & 7)) * 8]) = val;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < 64 * 8; e += blockDim.x) {
    const int cc = e >> 3, tch = e & 7;
    const int64_t t = t0 + tch * 8;
    if (t >= Tp) continue;
    // token rows tch * 8 .. + 7 all lie in row group tch
    const int col = (((cc >> 3) ^ tch) << 3) | (cc & 7);
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
      w[k] = static_cast<uint32_t>(tile[tch * 8 + 2 * k][col]) |
             (static_cast<uint32_t>(tile[tch * 8 + 2 * k + 1][col]) << 16);
    *reinterpret_cast<uint4*>(vt + (static_cast<int64_t>(g) * d + c0 + cc) * Tp + t) =
        make_uint4(w[0], w[1], w[2], w[3]);
  }
}

// ---------------------------------------------------------------- query tiles
// qtile_cu[r] = sum_{r' < r} ceil(T_r' / 128), one CTA.
__global__ void __launch_bounds__(1024)
k_attn_qtiles(const int32_t* __restrict__ cu, int R, int32_t* __restrict__ qtile_cu, const DevStatus* st) {
  __shared__ int32_t s_warp[32];
  __shared__ int32_t s_carry;
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (threadIdx.x == 0) s_carry = 0;
  __syncthreads();
  for (int base = 0; base < R; base += blockDim.x) {
    const int i = base + threadIdx.x;
    const int32_t v = i < R ? (cu[i + 1] - cu[i] + kQT - 1) / kQT : 0;
    int32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int32_t w = lane < nw ? s_warp[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int32_t y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      s_warp[lane] = w;
    }
    __syncthreads();
    const int32_t carry = s_carry;
    if (i < R) qtile_cu[i] = carry + (warp > 0 ? s_warp[warp - 1] : 0) + x - v;
    __syncthreads();
    if (threadIdx.x == 0) s_carry = carry + s_warp[nw - 1];
    __syncthreads();
  }
  if (threadIdx.x == 0) qtile_cu[R] = s_carry;
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

// A 3-D bf16 tensor map, 128-byte swizzle, box b0 x b1 x b2 (b0 * 2 bytes = 128).
bool map3(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t stride1_bytes,
          uint64_t stride2_bytes, uint32_t b0, uint32_t b1, uint32_t b2) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {b0, b1, b2};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_attn_forward(const avtp_layout_t& L, const avtp_score_args_t& sa, const avtp_forward_args_t& fa,
                                void* ws, const WsPlan& p, const FwdWs& f, cudaStream_t s) {
  if (L.n_tokens == 0) return cudaSuccess;
  static PerDevice attrs;
  cudaError_t e = once_per_device(attrs, [](int, int*) {
    return cudaFuncSetAttribute(k_attn_fwd, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kFwdSmem));
  });
  if (e != cudaSuccess) return e;
  const int d = sa.head_dim, Hq = sa.n_q_heads, Hkv = sa.n_kv_heads;
  const int64_t T = L.n_tokens, Tp = f.Tp;
  DevStatus* st = ws_at<DevStatus>(ws, p.status);
  __nv_bfloat16* vt = ws_at<__nv_bfloat16>(ws, f.vt);
  int32_t* qtile_cu = ws_at<int32_t>(ws, f.qtile_cu);

  e = launch_kernel(k_attn_qtiles, dim3(1), dim3(1024), 0, s, /*pdl=*/true, L.cu_seqlens, L.n_requests, qtile_cu,
                    static_cast<const DevStatus*>(st));
  if (e != cudaSuccess) return e;
  e = launch_kernel(k_attn_vt, dim3(static_cast<unsigned>((Tp + 63) / 64), d / 64, Hkv), dim3(256), 0, s,
                    /*pdl=*/true, static_cast<const __nv_bfloat16*>(fa.v), fa.v_stride, d, T, Tp, vt,
                    static_cast<const DevStatus*>(st));
  if (e != cudaSuccess) return e;

  CUtensorMap mq, mk, mv;
  if (!map3(&mq, sa.q, d, Hq, T, static_cast<uint64_t>(d) * 2, static_cast<uint64_t>(sa.q_stride) * 2, 64, 1, kQT) ||
      !map3(&mk, sa.k, d, Hkv, T, static_cast<uint64_t>(d) * 2, static_cast<uint64_t>(sa.k_stride) * 2, 64, 1, kKB) ||
      !map3(&mv, vt, Tp, d, Hkv, static_cast<uint64_t>(Tp) * 2, static_cast<uint64_t>(Tp) * d * 2, 64, d, 1))
    return cudaErrorInvalidValue;
  FwdArgs a{};
  a.cu = L.cu_seqlens;
  a.R = L.n_requests;
  a.qtile_cu = qtile_cu;
  a.Hq = Hq;
  a.G = Hq / Hkv;
  a.d = d;
  a.c2 = sa.softmax_scale * kLog2e;
  a.o = fa.o;
  a.o_stride = fa.o_stride;
  a.lse = fa.lse;
  a.lse_stride = fa.lse_stride;
  a.st = st;
  // query tiles: sum_r ceil(T_r / 128) <= T / 128 + R
  const int64_t tiles = T / kQT + L.n_requests;
  const int64_t grid = tiles * Hq;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  return launch_kernel(k_attn_fwd, dim3(static_cast<unsigned>(grid)), dim3(kThreads), kFwdSmem, s, /*pdl=*/true, mq,
                       mk, mv, a);
}

}  // namespace avtp

extern "C" avtp_status_t avtp_forward_timeline(int64_t* out, int32_t max_blocks) {
#ifdef AVTP_TIMELINE
  if (out == nullptr || max_blocks < 1) return AVTP_ERR_INVALID_ARG;
  const int n = max_blocks < avtp::kFwdTlBlocks ? max_blocks : avtp::kFwdTlBlocks;
  return cudaMemcpyFromSymbol(out, avtp::g_fwd_tl, static_cast<size_t>(n) * avtp::kFwdTlSlots * sizeof(long long)) ==
                 cudaSuccess
             ? AVTP_OK
             : AVTP_ERR_CUDA;
#else
  (void)out;
  (void)max_blocks;
  return AVTP_ERR_UNSUPPORTED;
#endif
}
