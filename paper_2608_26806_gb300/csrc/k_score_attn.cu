// Criterion B: text-to-visual attention mass per visual token (the per-token form of
// the attention quantity of paper §3.3.2), without materialising the attention matrix:
//   s_t = 1/(Hq*|Q_r|) * sum_h sum_{q in Q_r, pos q >= pos t} exp2(z2(h,q,t) - lse2(h,q)),
//   z2 = softmax_scale * log2(e) * q_h . k_{g(h)},  lse2 = log2 sum_{visible keys} exp2(z2).
//
// Rows: for KV group g, row o*G + j is text query o (in text order over the batch)
// with query head g*G + j. The text queries are first repacked by group into
// Qt[g][row][d] (k_attn_pack), so that both passes read them with TMA boxes.
//
// Pass 1 (skipped when the caller supplies FlashAttention's LSE): a work item is one
// tile of 128 rows of a request against one chunk of its keys; S = Q_rows K^T runs on
// the tensor cores (tcgen05.mma, 128 x 256 per step, fp32 accumulator in TMEM) and the
// epilogue warps keep an online (max, sum) per row; k_attn_merge then combines the
// chunks of every row into lse2 (a separate kernel: merging inside pass 1, in
// whichever item finished a tile last, piled the merges onto a few CTAs).
// Pass 2: a work item is one tile of 128 visual keys of an image; S^T = K_tile Qt^T
// over the rows of every text query after the image (all of them see every key of
// the image), 256 rows per step; each epilogue thread owns one key and sums
// exp2(z2 - lse2) over the rows.
// Finalize: sum the KV groups in a fixed order (deterministic), divide, and add the
// fixed-point per-image sums.
//
// Both passes are persistent (one CTA per SM). Warps 0-7 are the epilogue (warp w
// reads TMEM lanes 32(w%4)..+31, columns 128(w/4)..+127 of each step), warp 8 issues
// the TMA loads, warp 9 owns TMEM and issues the MMAs. Shared memory: two stages of
// A tiles (128 rows x d, so the next item's tile loads during this one) and two of
// B tiles (256 rows x d); TMEM: two 256-column accumulators, so the epilogue of one
// step overlaps the MMA of the next. The epilogue keeps four independent partial
// sums (and maxima) per thread: with two warps per scheduler there is little else
// to hide the latency of a dependent chain.
#include <cudaTypedefs.h>

#include "avtp_tc.cuh"

namespace avtp {
namespace {

constexpr int kM = kAttnTileM;   // 128
constexpr int kN = kAttnTileN;   // 256
constexpr int kEpiWarps = 8;     // warps 0-7: epilogue
constexpr int kTmaWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kThreads = 320;
constexpr uint32_t kTmemCols = 2 * kN;
constexpr float kLog2e = 1.4426950408889634f;

// Shared memory for head_dim d: two A stages, then two B stages, 1024-byte aligned.
__host__ __device__ constexpr size_t a_bytes(int d) { return static_cast<size_t>(kM) * d * 2; }
__host__ __device__ constexpr size_t b_bytes(int d) { return static_cast<size_t>(kN) * d * 2; }
__host__ __device__ constexpr size_t tc_smem_bytes(int d) { return 1024 + 2 * a_bytes(d) + 2 * b_bytes(d); }

struct Sync {
  uint64_t a_full[2], a_empty[2];
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
  const int32_t* img_req;
  const int32_t* text_idx;
  const int32_t* text_cu;
  const int32_t* qtile_cu;
  const int32_t* p1_cu;
  const int32_t* ktile_cu;
  float* lse_rows;        // [Hkv, rows]
  float2* p1_part;        // [Hkv * n_qtiles_max][128 rows][kAttnMaxChunks]
  float* partial;         // [Hkv, T]
  int64_t rows;           // rows per group
  int64_t p1_items_max;
  int G, Hkv, d, chunk_keys;
  float c2;               // softmax_scale * log2(e)
  DevStatus* st;
};

__device__ __forceinline__ void bar_epi() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

// ---------------------------------------------------------------- work items
struct P1Item {
  int g, qt, chunk;
  int64_t row0;      // first row (within group g) of the tile
  int64_t row_end;   // end of the request's rows, at most row0 + kM
  int key0, key_end; // packed key positions of the chunk
};

__device__ __forceinline__ P1Item p1_item(const AttnArgs& a, int n_per_group, int id) {
  P1Item it;
  it.g = id / n_per_group;
  const int rest = id - it.g * n_per_group;
  const int nq = a.qtile_cu[a.R];
  it.qt = upper_index(a.p1_cu, nq, rest);
  it.chunk = rest - a.p1_cu[it.qt];
  const int r = upper_index(a.qtile_cu, a.R, it.qt);
  const int64_t rr0 = static_cast<int64_t>(a.text_cu[r]) * a.G, rr1 = static_cast<int64_t>(a.text_cu[r + 1]) * a.G;
  it.row0 = rr0 + static_cast<int64_t>(it.qt - a.qtile_cu[r]) * kM;
  it.row_end = min(it.row0 + kM, rr1);
  const int pmax = a.text_idx[(it.row_end - 1) / a.G];
  it.key0 = a.cu[r] + it.chunk * a.chunk_keys;
  it.key_end = min(it.key0 + a.chunk_keys, pmax + 1);
  return it;
}

struct P2Item {
  int g, img;
  int kp0, nk;           // packed position of the tile's first key, keys in the tile
  int64_t row_begin, row_end;  // rows (within group g) of the text queries after the image
};

__device__ __forceinline__ P2Item p2_item(const AttnArgs& a, int n_per_group, int id) {
  P2Item it;
  it.g = id / n_per_group;
  const int b = id - it.g * n_per_group;
  const int i = upper_index(a.ktile_cu, a.NI, b);
  const int r = a.img_req[i];
  const int j = b - a.ktile_cu[i];
  it.img = i;
  it.kp0 = a.cu[r] + a.ist[i] + j * kM;
  it.nk = min(kM, a.iln[i] - j * kM);
  // text ordinal of the first token after the image: its request-local position minus the
  // visual tokens before it, plus the request's first text ordinal
  const int after = a.ist[i] + a.iln[i];
  const int o_first = a.text_cu[r] + after - (a.vis_cu[i + 1] - a.vis_cu[a.icu[r]]);
  it.row_begin = static_cast<int64_t>(o_first) * a.G;
  it.row_end = static_cast<int64_t>(a.text_cu[r + 1]) * a.G;
  return it;
}

// ---------------------------------------------------------------- the persistent kernel
// PASS 1: A = Qt rows (box 64 x 128), B = key tiles (box 64 x 256).
// PASS 2: A = key tile (box 64 x 128), B = Qt rows (box 64 x 256).
// Epilogue warp w reads TMEM lane quadrant w % 4 and column half w / 4 of each step.
template <int PASS>
__global__ void __launch_bounds__(kThreads, 1)
k_attn_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, AttnArgs a) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ Sync sy;
  __shared__ __align__(16) float s_lse[2][kN];
  __shared__ float2 s_mrg[2][kM];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int d = a.d;
  unsigned char* sA[2] = {smem, smem + a_bytes(d)};
  unsigned char* sB[2] = {smem + 2 * a_bytes(d), smem + 2 * a_bytes(d) + b_bytes(d)};
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t atomA = kM * 128, atomB = kN * 128;  // bytes per 64-element atom column

  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int n_per_group = (PASS == 1) ? a.p1_cu[a.qtile_cu[a.R]] : a.ktile_cu[a.NI];
  const int n_items = n_per_group * a.Hkv;
  if (static_cast<int>(blockIdx.x) >= n_items) return;

  if (threadIdx.x == 0) {
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&sy.a_full[s], 1);
      tc::mbar_init(&sy.a_empty[s], 1);
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
  const uint32_t tmem = sy.tmem;
  volatile int* abort_flag = &sy.abort;

  // B steps of an item (0: nothing to compute)
  auto item_steps = [&](int id, int& a_y, int& a_z, int64_t& b0) {
    if (PASS == 1) {
      const P1Item it = p1_item(a, n_per_group, id);
      a_y = static_cast<int>(it.row0);
      a_z = it.g;
      b0 = it.key0;
      return (it.key_end - it.key0 + kN - 1) / kN;
    }
    const P2Item it = p2_item(a, n_per_group, id);
    a_y = it.g;
    a_z = it.kp0;
    b0 = it.row_begin;
    return it.row_end > it.row_begin ? static_cast<int>((it.row_end - it.row_begin + kN - 1) / kN) : 0;
  };

  if (warp == kTmaWarp) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tc::tma_prefetch_map(&mapA);
      tc::tma_prefetch_map(&mapB);
      uint32_t na = 0, nb = 0;  // A loads and B loads issued so far
      for (int id = blockIdx.x; id < n_items && !*abort_flag; id += gridDim.x) {
        int a_y, a_z;
        int64_t b0;
        const int steps = item_steps(id, a_y, a_z, b0);
        if (steps <= 0) continue;
        const int sa = na & 1;
        if (na >= 2 && !tc::mbar_wait(&sy.a_empty[sa], ((na >> 1) - 1) & 1)) { *abort_flag = 1; break; }
        tc::mbar_arrive_expect_tx(&sy.a_full[sa], static_cast<uint32_t>(a_bytes(d)));
        for (int ac = 0; ac < d / 64; ++ac) tc::tma_load_3d(sA[sa] + ac * atomA, &mapA, ac * 64, a_y, a_z, &sy.a_full[sa]);
        ++na;
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          if (nb >= 2 && !tc::mbar_wait(&sy.b_empty[s], ((nb >> 1) - 1) & 1)) { *abort_flag = 1; break; }
          tc::mbar_arrive_expect_tx(&sy.b_full[s], static_cast<uint32_t>(b_bytes(d)));
          const int y = static_cast<int>(b0 + static_cast<int64_t>(st) * kN);
          for (int ac = 0; ac < d / 64; ++ac) {
            if (PASS == 1) tc::tma_load_3d(sB[s] + ac * atomB, &mapB, ac * 64, a_z, y, &sy.b_full[s]);  // {d, Hkv, T}
            else tc::tma_load_3d(sB[s] + ac * atomB, &mapB, ac * 64, y, a_y, &sy.b_full[s]);            // {d, rows, Hkv}
          }
        }
      }
      // let the copies in flight land before the CTA may exit
      for (uint32_t k = (na >= 2 ? na - 2 : 0); k < na; ++k) tc::mbar_wait(&sy.a_full[k & 1], (k >> 1) & 1);
      for (uint32_t k = (nb >= 2 ? nb - 2 : 0); k < nb; ++k) tc::mbar_wait(&sy.b_full[k & 1], (k >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(kM, kN);
      uint32_t na = 0, nb = 0;
      for (int id = blockIdx.x; id < n_items && !*abort_flag; id += gridDim.x) {
        int a_y, a_z;
        int64_t b0;
        const int steps = item_steps(id, a_y, a_z, b0);
        if (steps <= 0) continue;
        const int sa = na & 1;
        if (!tc::mbar_wait(&sy.a_full[sa], (na >> 1) & 1)) { *abort_flag = 1; break; }
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          if (!tc::mbar_wait(&sy.b_full[s], (nb >> 1) & 1)) { *abort_flag = 1; break; }
          if (nb >= 2 && !tc::mbar_wait(&sy.acc_empty[s], ((nb >> 1) - 1) & 1)) { *abort_flag = 1; break; }
          tc::fence_after_sync();
          tc::mma_rows(tmem + s * kN, tc::smem_u32(sA[sa]), atomA, tc::smem_u32(sB[s]), atomB, d, idesc);
          tc::mma_commit(&sy.b_empty[s]);
          tc::mma_commit(&sy.acc_full[s]);
        }
        tc::mma_commit(&sy.a_empty[sa]);
        ++na;
      }
      // every MMA issued has completed once this arrives
      tc::mma_commit(&sy.drain);
      tc::mbar_wait(&sy.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue (8 warps)
    const int etid = threadIdx.x;               // 0 .. 255
    const int quad = warp & 3, half = warp >> 2;
    const int lrow = quad * 32 + lane;          // TMEM lane: row (pass 1) or key (pass 2) of the tile
    const uint32_t taddr = tmem + (static_cast<uint32_t>(quad * 32) << 16) + half * (kN / 2);
    const float c2 = a.c2;
    // After a timeout (abort_flag) the epilogue keeps walking the same items and steps,
    // skipping every wait and TMEM read, so that its named barriers still line up.
    uint32_t nb = 0;
    int it_count = 0;
    for (int id = blockIdx.x; id < n_items; id += gridDim.x, ++it_count) {
      const int slot = it_count & 1;
      if (PASS == 1) {
        const P1Item it = p1_item(a, n_per_group, id);
        const int steps = (it.key_end - it.key0 + kN - 1) / kN;
        const int64_t row = it.row0 + lrow;
        const bool valid = row < it.row_end;
        const int qpos = valid ? a.text_idx[row / a.G] : -1;
        // keys up to min(qpos, key_end - 1) are visible to this row
        const int last = min(qpos, it.key_end - 1);
        float m = -INFINITY, l = 0.f;  // running max and sum, scaled (log2) domain
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          bool ok = !__any_sync(0xffffffffu, *abort_flag != 0);
          if (ok && !tc::mbar_wait_warp(&sy.acc_full[s], (nb >> 1) & 1)) {
            if (lane == 0) *abort_flag = 1;
            ok = false;
          }
          tc::fence_after_sync();
          const int k0 = it.key0 + st * kN + half * (kN / 2);  // key of this thread's first column
          const int lim = last - k0;                            // columns 0..lim are visible
          const bool all_visible = __all_sync(0xffffffffu, lim >= kN / 2 - 1);
          const bool any_visible = __any_sync(0xffffffffu, lim >= 0);
          if (ok && any_visible) {
#pragma unroll 1
            for (int p = 0; p < kN / 2 / 64; ++p) {
              float v[64];
              tc::tmem_ld64(taddr + s * kN + p * 64, v);
              if (!all_visible) {
#pragma unroll
                for (int q = 0; q < 64; ++q) v[q] = (p * 64 + q <= lim) ? v[q] : -INFINITY;
              }
              float mx0 = v[0], mx1 = v[1], mx2 = v[2], mx3 = v[3];
#pragma unroll
              for (int q = 4; q < 64; q += 4) {
                mx0 = fmaxf(mx0, v[q]);
                mx1 = fmaxf(mx1, v[q + 1]);
                mx2 = fmaxf(mx2, v[q + 2]);
                mx3 = fmaxf(mx3, v[q + 3]);
              }
              const float mn = fmaxf(m, fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * c2);
              if (mn != -INFINITY) {
                float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
                for (int q = 0; q < 64; q += 4) {
                  s0 += tc::ex2(fmaf(v[q], c2, -mn));
                  s1 += tc::ex2(fmaf(v[q + 1], c2, -mn));
                  s2 += tc::ex2(fmaf(v[q + 2], c2, -mn));
                  s3 += tc::ex2(fmaf(v[q + 3], c2, -mn));
                }
                l = l * tc::ex2(m - mn) + ((s0 + s1) + (s2 + s3));
                m = mn;
              }
            }
          }
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(&sy.acc_empty[s]);
        }
        // the two column halves of a row meet here; this chunk's (max, sum) per row goes
        // to [row tile][row][chunk] for k_attn_merge
        if (half == 1) s_mrg[slot][lrow] = make_float2(m, l);
        bar_epi();
        if (half == 0) {
          const float2 o = s_mrg[slot][lrow];
          const float M = fmaxf(m, o.x);
          const float L = (M == -INFINITY) ? 0.f : l * tc::ex2(m - M) + o.y * tc::ex2(o.x - M);
          const int64_t tile = static_cast<int64_t>(it.g) * a.qtile_cu[a.R] + it.qt;
          a.p1_part[(tile * kM + lrow) * kAttnMaxChunks + it.chunk] = make_float2(M, L);
        }
      } else {
        const P2Item it = p2_item(a, n_per_group, id);
        const int steps =
            it.row_end > it.row_begin ? static_cast<int>((it.row_end - it.row_begin + kN - 1) / kN) : 0;
        const float* lse_g = a.lse_rows + static_cast<int64_t>(it.g) * a.rows;
        // the rows' lse2 (+inf past the last row, which zeroes their terms); the next
        // step's value is loaded while this step is processed
        auto lse_of = [&](int st) {
          const int64_t r = it.row_begin + static_cast<int64_t>(st) * kN + etid;
          return (st < steps && r < it.row_end) ? lse_g[r] : INFINITY;
        };
        float lse_next = lse_of(0);
        float m0 = 0.f, m1 = 0.f, m2 = 0.f, m3 = 0.f;
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          s_lse[s][etid] = lse_next;
          bar_epi();
          lse_next = lse_of(st + 1);
          bool ok = !__any_sync(0xffffffffu, *abort_flag != 0);
          if (ok && !tc::mbar_wait_warp(&sy.acc_full[s], (nb >> 1) & 1)) {
            if (lane == 0) *abort_flag = 1;
            ok = false;
          }
          tc::fence_after_sync();
#pragma unroll 1
          for (int p = 0; p < (ok ? kN / 2 / 64 : 0); ++p) {
            float v[64];
            tc::tmem_ld64(taddr + s * kN + p * 64, v);
            const float4* l4 = reinterpret_cast<const float4*>(&s_lse[s][half * (kN / 2) + p * 64]);
#pragma unroll
            for (int q4 = 0; q4 < 16; ++q4) {
              const float4 lv = l4[q4];
              m0 += tc::ex2(fmaf(v[4 * q4 + 0], c2, -lv.x));
              m1 += tc::ex2(fmaf(v[4 * q4 + 1], c2, -lv.y));
              m2 += tc::ex2(fmaf(v[4 * q4 + 2], c2, -lv.z));
              m3 += tc::ex2(fmaf(v[4 * q4 + 3], c2, -lv.w));
            }
          }
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(&sy.acc_empty[s]);
        }
        const float mass = (m0 + m1) + (m2 + m3);
        if (half == 1) s_mrg[slot][lrow].x = mass;
        bar_epi();
        if (half == 0 && lrow < it.nk)
          a.partial[static_cast<int64_t>(it.g) * a.T + it.kp0 + lrow] = mass + s_mrg[slot][lrow].x;
      }
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

// ---------------------------------------------------------------- pass-1 chunk merge
// lse2 of every row: the log2-sum-exp2 merge of its chunks' (max, sum). One thread per
// (KV group, row); a row's chunks are contiguous.
__global__ void __launch_bounds__(256)
k_attn_merge(AttnArgs a) {
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int nq = a.qtile_cu[a.R];
  const int64_t total = static_cast<int64_t>(a.Hkv) * nq * kM;
  for (int64_t u = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; u < total;
       u += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int lr = static_cast<int>(u % kM);
    const int64_t tile = u / kM;
    const int g = static_cast<int>(tile / nq), qt = static_cast<int>(tile - static_cast<int64_t>(g) * nq);
    const int r = upper_index(a.qtile_cu, a.R, qt);
    const int64_t row = static_cast<int64_t>(a.text_cu[r]) * a.G + static_cast<int64_t>(qt - a.qtile_cu[r]) * kM + lr;
    if (row >= static_cast<int64_t>(a.text_cu[r + 1]) * a.G) continue;
    const int nc = a.p1_cu[qt + 1] - a.p1_cu[qt];
    const float4* src = reinterpret_cast<const float4*>(a.p1_part + u * kAttnMaxChunks);
    float M = -INFINITY, L = 0.f;
    auto merge = [&](float mc, float lc) {
      const float Mn = fmaxf(M, mc);
      if (Mn != -INFINITY) {
        L = L * tc::ex2(M - Mn) + lc * tc::ex2(mc - Mn);
        M = Mn;
      }
    };
    const int n4 = (nc + 1) >> 1;  // a float4 holds two chunks
    for (int c4 = 0; c4 < n4; c4 += 8) {
      float4 buf[8];
#pragma unroll
      for (int w = 0; w < 8; ++w)
        buf[w] = (c4 + w < n4) ? __ldg(src + c4 + w) : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        merge(buf[w].x, buf[w].y);
        if (2 * (c4 + w) + 1 < nc) merge(buf[w].z, buf[w].w);
      }
    }
    a.lse_rows[static_cast<int64_t>(g) * a.rows + row] = M + __log2f(L);
  }
}

// ---------------------------------------------------------------- repacking of the text queries
// Qt[g][o*G + j][:] = q[text_idx[o], g*G + j, :]; with a supplied LSE also
// lse_rows[g][o*G + j] = lse[g*G + j][text_idx[o]] * log2(e). One thread per 16 bytes.
__global__ void __launch_bounds__(256)
k_attn_pack(const __nv_bfloat16* __restrict__ q, int64_t q_stride, int Hq, int G, int d,
            const int32_t* __restrict__ text_idx, const int32_t* __restrict__ text_cu, int R, int64_t rows,
            __nv_bfloat16* __restrict__ qt, const float* __restrict__ lse, int64_t lse_stride,
            float* __restrict__ lse_rows, const DevStatus* st) {
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int64_t n_text = text_cu[R];
  const int vec = d / 8;
  const int64_t total = n_text * Hq * vec;
  for (int64_t u = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; u < total;
       u += static_cast<int64_t>(gridDim.x) * blockDim.x) {
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
__global__ void __launch_bounds__(256)
k_attn_finalize(const float* __restrict__ partial, int Hq, int Hkv, int64_t T, const int32_t* __restrict__ cu,
                const int32_t* __restrict__ img_start, const int32_t* __restrict__ vis_cu,
                const int32_t* __restrict__ img_req, const int32_t* __restrict__ text_cu, int NI,
                float* __restrict__ scores, int64_t* __restrict__ img_sums, const DevStatus* st) {
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int n_vis = vis_cu[NI];
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < n_vis;
       v += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = upper_index(vis_cu, NI, v);
    const int r = img_req[i];
    const int64_t t = static_cast<int64_t>(cu[r]) + img_start[i] + (v - vis_cu[i]);
    const int nq = text_cu[r + 1] - text_cu[r];
    float s = 0.f;
    if (nq > 0) {
      for (int g = 0; g < Hkv; ++g) s += partial[static_cast<int64_t>(g) * T + t];
      s = s / static_cast<float>(static_cast<int64_t>(Hq) * nq);
    }
    scores[t] = s;
    atomicAdd(reinterpret_cast<unsigned long long*>(img_sums + i), static_cast<unsigned long long>(fixed_point_score(s)));
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
  static bool attr_set[2] = {false, false};
  const size_t smem = tc_smem_bytes(d);
  const int di = d == 128 ? 1 : 0;
  if (!attr_set[di]) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_tc<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(tc_smem_bytes(128)));
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_attn_tc<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(tc_smem_bytes(128)));
    if (e != cudaSuccess) return e;
    attr_set[0] = attr_set[1] = true;
  }
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
  a.img_req = ws_at<int32_t>(ws, p.img_req);
  a.text_idx = ws_at<int32_t>(ws, p.text_idx);
  a.text_cu = ws_at<int32_t>(ws, p.text_cu);
  a.qtile_cu = ws_at<int32_t>(ws, p.qtile_cu);
  a.p1_cu = ws_at<int32_t>(ws, p.p1_cu);
  a.ktile_cu = ws_at<int32_t>(ws, p.ktile_cu);
  a.lse_rows = ws_at<float>(ws, p.lse_rows);
  a.p1_part = sa.lse == nullptr ? ws_at<float2>(ws, p.p1_part) : nullptr;
  a.partial = ws_at<float>(ws, p.partial);
  a.rows = plan.rows;
  a.p1_items_max = plan.p1_items_max;
  a.G = plan.G;
  a.Hkv = Hkv;
  a.d = d;
  a.chunk_keys = plan.chunk_keys;
  a.c2 = sa.softmax_scale * kLog2e;
  a.st = st;
  __nv_bfloat16* qt = ws_at<__nv_bfloat16>(ws, p.qt);

  // tensor maps: keys {d, Hkv, T} (token stride k_stride), packed queries {d, rows, Hkv}
  CUtensorMap mk128, mk256, mq128, mq256;
  const uint64_t ks = static_cast<uint64_t>(sa.k_stride) * 2, qs = static_cast<uint64_t>(plan.rows) * d * 2;
  if (!make_map(&mk128, sa.k, d, Hkv, L.n_tokens, static_cast<uint64_t>(d) * 2, ks, 1, kM) ||
      !make_map(&mk256, sa.k, d, Hkv, L.n_tokens, static_cast<uint64_t>(d) * 2, ks, 1, kN) ||
      !make_map(&mq128, qt, d, plan.rows, Hkv, static_cast<uint64_t>(d) * 2, qs, kM, 1) ||
      !make_map(&mq256, qt, d, plan.rows, Hkv, static_cast<uint64_t>(d) * 2, qs, kN, 1))
    return cudaErrorInvalidValue;

  const int sms = device_sm_count();
  {
    const int64_t want = (plan.max_text * Hq * (d / 8) + 255) / 256;
    const int64_t cap = static_cast<int64_t>(sms) * 8;
    const int grid = static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
    cudaError_t e = launch_kernel(k_attn_pack, dim3(grid), dim3(256), 0, s, /*pdl=*/true,
                                  static_cast<const __nv_bfloat16*>(sa.q), sa.q_stride, Hq, plan.G, d, a.text_idx,
                                  a.text_cu, L.n_requests, plan.rows, qt, sa.lse, sa.lse_stride, a.lse_rows,
                                  static_cast<const DevStatus*>(st));
    if (e != cudaSuccess) return e;
  }
  if (sa.lse == nullptr) {
    cudaError_t e = launch_kernel(k_attn_tc<1>, dim3(sms), dim3(kThreads), smem, s, /*pdl=*/true, mq128, mk256, a);
    if (e != cudaSuccess) return e;
    const int64_t rows_max = static_cast<int64_t>(Hkv) * plan.n_qtiles_max * kM;
    const int64_t cap = static_cast<int64_t>(sms) * 4;
    const int64_t want = (rows_max + 255) / 256;
    e = launch_kernel(k_attn_merge, dim3(static_cast<unsigned>(want < cap ? want : cap)), dim3(256), 0, s,
                      /*pdl=*/true, a);
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = launch_kernel(k_attn_tc<2>, dim3(sms), dim3(kThreads), smem, s, /*pdl=*/true, mk128, mq256, a);
  if (e != cudaSuccess) return e;
  const int64_t want = (L.n_tokens + 255) / 256;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  const int grid3 = static_cast<int>(want < cap ? want : cap);
  return launch_kernel(k_attn_finalize, dim3(grid3), dim3(256), 0, s, /*pdl=*/true, a.partial, Hq, Hkv, L.n_tokens,
                       L.cu_seqlens, L.img_start, a.vis_cu, a.img_req, a.text_cu, L.n_images, scores, img_sums,
                       static_cast<const DevStatus*>(st));
}

}  // namespace avtp
