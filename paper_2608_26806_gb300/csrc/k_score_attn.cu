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
// epilogue warps keep an online (max, sum) per row. The last item of a tile merges
// the chunks into lse2.
// Pass 2: a work item is one tile of 128 visual keys of an image; S^T = K_tile Qt^T
// over the rows of every text query after the image (all of them see every key of
// the image), 256 rows per step; each epilogue thread owns one key and sums
// exp2(z2 - lse2) over the rows.
// Finalize: sum the KV groups in a fixed order (deterministic), divide, and add the
// fixed-point per-image sums.
//
// Both passes are persistent (one CTA per SM). Warps 0-3 are the epilogue (warp w
// reads TMEM lanes 32w..32w+31), warp 4 issues the TMA loads, warp 5 owns TMEM and
// issues the MMAs. Shared memory: the item's A tile (128 rows x d) and two stages of
// B tiles (256 rows x d); TMEM: two 256-column accumulators, so the epilogue of one
// step overlaps the MMA of the next.
#include <cudaTypedefs.h>

#include "avtp_tc.cuh"

namespace avtp {
namespace {

constexpr int kM = kAttnTileM;   // 128
constexpr int kN = kAttnTileN;   // 256
constexpr int kThreads = 192;
constexpr int kEpiThreads = 128;
constexpr uint32_t kTmemCols = 2 * kN;
constexpr float kLog2e = 1.4426950408889634f;

// Shared memory for head_dim d: A tile, then two B stages, 1024-byte aligned.
__host__ __device__ constexpr size_t a_bytes(int d) { return static_cast<size_t>(kM) * d * 2; }
__host__ __device__ constexpr size_t b_bytes(int d) { return static_cast<size_t>(kN) * d * 2; }
__host__ __device__ constexpr size_t tc_smem_bytes(int d) { return 1024 + a_bytes(d) + 2 * b_bytes(d); }

struct Sync {
  uint64_t a_full, a_empty;
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
  int32_t* p1_cnt;
  const int32_t* ktile_cu;
  float* lse_rows;        // [Hkv, rows]
  float2* p1_part;        // [Hkv * p1_items_max * 128]
  float* partial;         // [Hkv, T]
  int64_t rows;           // rows per group
  int64_t p1_items_max;
  int G, Hkv, d, chunk_keys;
  float c2;               // softmax_scale * log2(e)
  DevStatus* st;
};

__device__ __forceinline__ void bar_epi() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

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
// PASS 1: A = Qt rows (map qa, box 64 x 128), B = key tiles (map kb, box 64 x 256).
// PASS 2: A = key tile (map ka, box 64 x 128), B = Qt rows (map qb, box 64 x 256).
template <int PASS>
__global__ void __launch_bounds__(kThreads, 1)
k_attn_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, AttnArgs a) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ Sync sy;
  __shared__ float s_lse[2][kN];
  __shared__ int s_last;
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* sA = smem;
  unsigned char* sB[2] = {smem + a_bytes(a.d), smem + a_bytes(a.d) + b_bytes(a.d)};
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d = a.d;
  const uint32_t atomA = kM * 128, atomB = kN * 128;  // bytes per 64-element atom column

  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  int n_per_group;
  if (PASS == 1) {
    n_per_group = a.p1_cu[a.qtile_cu[a.R]];
  } else {
    n_per_group = a.ktile_cu[a.NI];
  }
  const int n_items = n_per_group * a.Hkv;
  if (static_cast<int>(blockIdx.x) >= n_items) return;

  if (threadIdx.x == 0) {
    tc::mbar_init(&sy.a_full, 1);
    tc::mbar_init(&sy.a_empty, 1);
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&sy.b_full[s], 1);
      tc::mbar_init(&sy.b_empty[s], 1);
      tc::mbar_init(&sy.acc_full[s], 1);
      tc::mbar_init(&sy.acc_empty[s], kEpiThreads / 32);
    }
    tc::mbar_init(&sy.drain, 1);
    sy.abort = 0;
    tc::fence_mbar_init();
  }
  if (warp == 5) {
    tc::tmem_alloc(&sy.tmem, kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sy.tmem;
  volatile int* abort_flag = &sy.abort;

  if (warp == 4) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tc::tma_prefetch_map(&mapA);
      tc::tma_prefetch_map(&mapB);
      uint32_t na = 0, nb = 0;  // A loads and B loads issued so far
      for (int id = blockIdx.x; id < n_items && !*abort_flag; id += gridDim.x) {
        int a_y, a_z, steps;
        int64_t b0;  // first B row of the item (key position or row index)
        if (PASS == 1) {
          const P1Item it = p1_item(a, n_per_group, id);
          a_y = static_cast<int>(it.row0);
          a_z = it.g;
          b0 = it.key0;
          steps = (it.key_end - it.key0 + kN - 1) / kN;
        } else {
          const P2Item it = p2_item(a, n_per_group, id);
          a_y = it.g;
          a_z = it.kp0;
          b0 = it.row_begin;
          steps = it.row_end > it.row_begin ? static_cast<int>((it.row_end - it.row_begin + kN - 1) / kN) : 0;
        }
        if (steps <= 0) continue;
        if (na > 0 && !tc::mbar_wait(&sy.a_empty, (na - 1) & 1)) { *abort_flag = 1; break; }
        tc::mbar_arrive_expect_tx(&sy.a_full, static_cast<uint32_t>(a_bytes(d)));
        for (int ac = 0; ac < d / 64; ++ac) tc::tma_load_3d(sA + ac * atomA, &mapA, ac * 64, a_y, a_z, &sy.a_full);
        ++na;
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          if (nb >= 2 && !tc::mbar_wait(&sy.b_empty[s], ((nb >> 1) - 1) & 1)) { *abort_flag = 1; break; }
          tc::mbar_arrive_expect_tx(&sy.b_full[s], static_cast<uint32_t>(b_bytes(d)));
          const int64_t y = b0 + static_cast<int64_t>(st) * kN;
          for (int ac = 0; ac < d / 64; ++ac) {
            if (PASS == 1) {  // keys: map dims {d, Hkv, T}
              tc::tma_load_3d(sB[s] + ac * atomB, &mapB, ac * 64, a_z, static_cast<int>(y), &sy.b_full[s]);
            } else {          // rows: map dims {d, rows, Hkv}
              tc::tma_load_3d(sB[s] + ac * atomB, &mapB, ac * 64, static_cast<int>(y), a_y, &sy.b_full[s]);
            }
          }
        }
      }
      // let the copies in flight land before the CTA may exit
      if (na > 0) tc::mbar_wait(&sy.a_full, (na - 1) & 1);
      for (uint32_t k = (nb >= 2 ? nb - 2 : 0); k < nb; ++k) tc::mbar_wait(&sy.b_full[k & 1], (k >> 1) & 1);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(kM, kN);
      uint32_t na = 0, nb = 0;
      for (int id = blockIdx.x; id < n_items && !*abort_flag; id += gridDim.x) {
        int steps;
        if (PASS == 1) {
          const P1Item it = p1_item(a, n_per_group, id);
          steps = (it.key_end - it.key0 + kN - 1) / kN;
        } else {
          const P2Item it = p2_item(a, n_per_group, id);
          steps = it.row_end > it.row_begin ? static_cast<int>((it.row_end - it.row_begin + kN - 1) / kN) : 0;
        }
        if (steps <= 0) continue;
        if (!tc::mbar_wait(&sy.a_full, na & 1)) { *abort_flag = 1; break; }
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          if (!tc::mbar_wait(&sy.b_full[s], (nb >> 1) & 1)) { *abort_flag = 1; break; }
          if (nb >= 2 && !tc::mbar_wait(&sy.acc_empty[s], ((nb >> 1) - 1) & 1)) { *abort_flag = 1; break; }
          tc::fence_after_sync();
          tc::mma_rows(tmem + s * kN, tc::smem_u32(sA), atomA, tc::smem_u32(sB[s]), atomB, d, idesc);
          tc::mma_commit(&sy.b_empty[s]);
          tc::mma_commit(&sy.acc_full[s]);
        }
        tc::mma_commit(&sy.a_empty);
        ++na;
      }
      // every MMA issued has completed once this arrives
      tc::mma_commit(&sy.drain);
      tc::mbar_wait(&sy.drain, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue (128 threads)
    const int etid = threadIdx.x;                       // 0..127 = TMEM lane
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    uint32_t nb = 0;
    for (int id = blockIdx.x; id < n_items && !*abort_flag; id += gridDim.x) {
      if (PASS == 1) {
        const P1Item it = p1_item(a, n_per_group, id);
        const int steps = (it.key_end - it.key0 + kN - 1) / kN;
        const int64_t row = it.row0 + etid;
        const bool valid = row < it.row_end;
        const int qpos = valid ? a.text_idx[row / a.G] : -1;
        // keys k0 + j with k0 + j <= min(qpos, key_end - 1) are visible to this row
        const int last = min(qpos, it.key_end - 1);
        float m = -INFINITY, l = 0.f;
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          if (!tc::mbar_wait_warp(&sy.acc_full[s], (nb >> 1) & 1)) { *abort_flag = 1; break; }
          tc::fence_after_sync();
          const int k0 = it.key0 + st * kN;
          const int lim = last - k0;  // columns 0..lim are visible
#pragma unroll 1
          for (int p = 0; p < kN / 32; ++p) {
            float v[32];
            tc::tmem_ld32(lane_addr + s * kN + p * 32, v);
            float pm = -INFINITY;
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              v[q] = (p * 32 + q <= lim) ? v[q] * a.c2 : -INFINITY;
              pm = fmaxf(pm, v[q]);
            }
            const float mn = fmaxf(m, pm);
            if (mn != -INFINITY) {
              float sum = 0.f;
#pragma unroll
              for (int q = 0; q < 32; ++q) sum += tc::ex2(v[q] - mn);
              l = l * tc::ex2(m - mn) + sum;
              m = mn;
            }
          }
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(&sy.acc_empty[s]);
        }
        if (*abort_flag) break;
        // this chunk's (max, sum) per row; the last chunk of the tile merges them
        const int64_t slot = (static_cast<int64_t>(id) * kM + etid);
        a.p1_part[slot] = make_float2(m, l);
        __threadfence();
        bar_epi();
        if (etid == 0) {
          const int nq = a.qtile_cu[a.R];
          const int nc = a.p1_cu[it.qt + 1] - a.p1_cu[it.qt];
          const int prev = atomicAdd(&a.p1_cnt[it.g * nq + it.qt], 1);
          s_last = (prev == nc - 1) ? 1 : 0;
          if (s_last) a.p1_cnt[it.g * nq + it.qt] = 0;  // ready for the next call
        }
        bar_epi();
        if (s_last) {
          __threadfence();
          const int nc = a.p1_cu[it.qt + 1] - a.p1_cu[it.qt];
          const int id0 = it.g * n_per_group + a.p1_cu[it.qt];
          float M = -INFINITY;
          for (int c = 0; c < nc; ++c) M = fmaxf(M, __ldcg(&a.p1_part[(static_cast<int64_t>(id0) + c) * kM + etid]).x);
          float L = 0.f;
          if (M != -INFINITY) {
            for (int c = 0; c < nc; ++c) {
              const float2 ml = __ldcg(&a.p1_part[(static_cast<int64_t>(id0) + c) * kM + etid]);
              if (ml.x != -INFINITY) L += ml.y * tc::ex2(ml.x - M);
            }
          }
          if (valid) a.lse_rows[static_cast<int64_t>(it.g) * a.rows + row] = M + __log2f(L);
        }
      } else {
        const P2Item it = p2_item(a, n_per_group, id);
        const int steps =
            it.row_end > it.row_begin ? static_cast<int>((it.row_end - it.row_begin + kN - 1) / kN) : 0;
        const float* lse_g = a.lse_rows + static_cast<int64_t>(it.g) * a.rows;
        float mass = 0.f;
        for (int st = 0; st < steps; ++st, ++nb) {
          const int s = nb & 1;
          // the rows' lse2 (+inf past the last row, which zeroes their terms)
          const int64_t r0 = it.row_begin + static_cast<int64_t>(st) * kN;
#pragma unroll
          for (int h = 0; h < kN / kEpiThreads; ++h) {
            const int j = etid + h * kEpiThreads;
            s_lse[s][j] = (r0 + j < it.row_end) ? lse_g[r0 + j] : INFINITY;
          }
          bar_epi();
          if (!tc::mbar_wait_warp(&sy.acc_full[s], (nb >> 1) & 1)) { *abort_flag = 1; break; }
          tc::fence_after_sync();
#pragma unroll 1
          for (int p = 0; p < kN / 32; ++p) {
            float v[32];
            tc::tmem_ld32(lane_addr + s * kN + p * 32, v);
            const float4* l4 = reinterpret_cast<const float4*>(&s_lse[s][p * 32]);
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
              const float4 lv = l4[q4];
              mass += tc::ex2(fmaf(v[4 * q4 + 0], a.c2, -lv.x));
              mass += tc::ex2(fmaf(v[4 * q4 + 1], a.c2, -lv.y));
              mass += tc::ex2(fmaf(v[4 * q4 + 2], a.c2, -lv.z));
              mass += tc::ex2(fmaf(v[4 * q4 + 3], a.c2, -lv.w));
            }
          }
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(&sy.acc_empty[s]);
        }
        if (*abort_flag) break;
        if (etid < it.nk) a.partial[static_cast<int64_t>(it.g) * a.T + it.kp0 + etid] = mass;
      }
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 5) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && sy.abort) record_error(a.st, AVTP_ERR_TIMEOUT, static_cast<int32_t>(blockIdx.x));
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
  a.p1_cnt = ws_at<int32_t>(ws, p.p1_cnt);
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
