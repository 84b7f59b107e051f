// Criterion B: text-to-visual attention mass per visual token (the per-token form
// of the attention quantity of paper §3.3.2), without materialising the
// attention matrix:
//   s_t = 1/(Hq*|Q_r|) * sum_h sum_{q in Q_r, pos q >= pos t} exp2(z2(h,q,t) - lse2(h,q)),
//   z2 = softmax_scale * log2(e) * q_h . k_{g(h)},  lse2 = log2 sum_{visible keys} exp2(z2).
//
// Pass 1 (skipped when the caller supplies FlashAttention's LSE): per (KV group,
// tile of text queries) stream the request's keys with an online max/sum.
// Pass 2: per (KV group, tile of 64 visual keys) stream the request's text queries
// that can see the tile and accumulate exp2(z2 - lse2) per key.
// Finalize: sum the KV groups in a fixed order (deterministic), divide, and add
// the fixed-point per-image sums.
//
// This file is the CUDA-core (fp32 FMA) path: tiles of 64 rows x 64 keys in
// shared memory, 16 products per thread.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kThreads = 256;
constexpr int kKT = kAttnKeyTile;   // 64 keys per tile
constexpr int kRows = kAttnRowTile; // 64 (head, query) rows per tile
constexpr float kLog2e = 1.4426950408889634f;

// Load `rows` rows of `d` bf16 (row r at src + r_off[r]) into fp32 shared memory with pitch d+1.
__device__ __forceinline__ void load_rows_f32(float* dst, const __nv_bfloat16* const* src_rows, int n_rows,
                                              int d) {
  const int vec_per_row = d >> 3;
  for (int v = threadIdx.x; v < kRows * vec_per_row; v += kThreads) {
    const int r = v / vec_per_row, c = (v % vec_per_row) * 8;
    float* o = dst + r * (d + 1) + c;
    if (r < n_rows && src_rows[r] != nullptr) {
      const uint4 raw = *reinterpret_cast<const uint4*>(src_rows[r] + c);
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(h[j]);
        o[2 * j] = f.x;
        o[2 * j + 1] = f.y;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) o[j] = 0.f;
    }
  }
}

// ---------------------------------------------------------------- pass 1: LSE
__global__ void __launch_bounds__(kThreads)
k_attn_lse(const __nv_bfloat16* __restrict__ q, int64_t q_stride, const __nv_bfloat16* __restrict__ k,
           int64_t k_stride, int Hq, int Hkv, int d, float c2, const int32_t* __restrict__ cu, int R,
           const int32_t* __restrict__ text_idx, const int32_t* __restrict__ text_cu,
           const int32_t* __restrict__ qtile_cu, int q_tile, float* __restrict__ lse2, int64_t T,
           const DevStatus* st) {
  extern __shared__ __align__(16) float sm[];
  __shared__ const __nv_bfloat16* s_rows[kRows];
  __shared__ int32_t s_rpos[kRows];
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int b = blockIdx.x, g = blockIdx.y;
  if (b >= qtile_cu[R]) return;
  const int r = upper_index(qtile_cu, R, b);
  const int G = Hq / Hkv;
  const int o0 = text_cu[r] + (b - qtile_cu[r]) * q_tile;
  const int nq = min(q_tile, text_cu[r + 1] - o0);
  const int n_rows = G * q_tile;  // <= kRows
  float* Qs = sm;
  float* Ks = sm + kRows * (d + 1);
  const int tid = threadIdx.x;
  if (tid < kRows) {
    const int hh = tid / q_tile, qi = tid % q_tile;
    if (tid < n_rows && qi < nq) {
      const int pos = text_idx[o0 + qi];
      s_rows[tid] = q + static_cast<int64_t>(pos) * q_stride + static_cast<int64_t>(g * G + hh) * d;
      s_rpos[tid] = pos;
    } else {
      s_rows[tid] = nullptr;
      s_rpos[tid] = -1;
    }
  }
  __syncthreads();
  load_rows_f32(Qs, s_rows, kRows, d);
  const int pmax = text_idx[o0 + nq - 1];
  const int ty = tid >> 4, tx = tid & 15;  // rows ty*4..+3, keys tx + 16*c
  float m_run[4], l_run[4];
  int rpos[4];
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    m_run[a] = -INFINITY;
    l_run[a] = 0.f;
    rpos[a] = s_rpos[ty * 4 + a];
  }
  __shared__ const __nv_bfloat16* s_keys[kKT];
  for (int k0 = cu[r]; k0 <= pmax; k0 += kKT) {
    __syncthreads();
    if (tid < kKT) {
      const int key = k0 + tid;
      s_keys[tid] = (key <= pmax) ? k + static_cast<int64_t>(key) * k_stride + static_cast<int64_t>(g) * d : nullptr;
    }
    __syncthreads();
    load_rows_f32(Ks, s_keys, kKT, d);
    __syncthreads();
    float acc[4][4] = {};
    for (int e = 0; e < d; ++e) {
      float qa[4], kb[4];
#pragma unroll
      for (int a = 0; a < 4; ++a) qa[a] = Qs[(ty * 4 + a) * (d + 1) + e];
#pragma unroll
      for (int c = 0; c < 4; ++c) kb[c] = Ks[(tx + 16 * c) * (d + 1) + e];
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a][c] = fmaf(qa[a], kb[c], acc[a][c]);
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      float z[4];
      float mt = -INFINITY;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int key = k0 + tx + 16 * c;
        z[c] = (rpos[a] >= 0 && key <= rpos[a]) ? acc[a][c] * c2 : -INFINITY;
        mt = fmaxf(mt, z[c]);
      }
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
      const float mn = fmaxf(m_run[a], mt);
      const bool any = mn != -INFINITY;  // uniform over the 16 lanes of this row
      float ls = 0.f;
#pragma unroll
      for (int c = 0; c < 4; ++c) ls += any ? exp2f(z[c] - mn) : 0.f;
      // every lane takes part in the shuffles, whatever its row's state
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o);
      if (any) {
        l_run[a] = l_run[a] * exp2f(m_run[a] - mn) + ls;
        m_run[a] = mn;
      }
    }
  }
  if (tx == 0) {
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int row = ty * 4 + a;
      if (rpos[a] >= 0) {
        const int hh = row / q_tile;
        lse2[static_cast<int64_t>(g * G + hh) * T + rpos[a]] = m_run[a] + log2f(l_run[a]);
      }
    }
  }
}

// ---------------------------------------------------------------- pass 2: probability mass per key
__global__ void __launch_bounds__(kThreads)
k_attn_mass(const __nv_bfloat16* __restrict__ q, int64_t q_stride, const __nv_bfloat16* __restrict__ k,
            int64_t k_stride, int Hq, int Hkv, int d, float c2, const int32_t* __restrict__ cu,
            const int32_t* __restrict__ img_start, const int32_t* __restrict__ img_len,
            const int32_t* __restrict__ img_req, int NI, const int32_t* __restrict__ text_idx,
            const int32_t* __restrict__ text_cu, const int32_t* __restrict__ ktile_cu, int q_tile,
            const float* __restrict__ lse, int64_t lse_stride, float lse_mul, float* __restrict__ partial, int64_t T,
            const DevStatus* st) {
  extern __shared__ __align__(16) float sm[];
  __shared__ const __nv_bfloat16* s_rows[kRows];
  __shared__ const __nv_bfloat16* s_keys[kKT];
  __shared__ int32_t s_rpos[kRows];
  __shared__ float s_rlse[kRows];
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int b = blockIdx.x, g = blockIdx.y;
  if (b >= ktile_cu[NI]) return;
  const int i = upper_index(ktile_cu, NI, b);
  const int r = img_req[i];
  const int G = Hq / Hkv;
  const int j0 = (b - ktile_cu[i]) * kKT;
  const int nk = min(kKT, img_len[i] - j0);
  const int kp0 = cu[r] + img_start[i] + j0;  // packed position of the tile's first key
  float* Ks = sm;
  float* Qs = sm + kKT * (d + 1);
  const int tid = threadIdx.x;
  if (tid < kKT)
    s_keys[tid] = (tid < nk) ? k + static_cast<int64_t>(kp0 + tid) * k_stride + static_cast<int64_t>(g) * d : nullptr;
  __syncthreads();
  load_rows_f32(Ks, s_keys, kKT, d);
  // first text query of request r that can see the tile's first key (pos >= kp0)
  int lo = text_cu[r], hi = text_cu[r + 1];
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (text_idx[mid] < kp0) lo = mid + 1; else hi = mid;
  }
  const int o_end = text_cu[r + 1];
  const int ty = tid >> 4, tx = tid & 15;  // keys ty*4..+3, rows tx + 16*c
  float mass[4] = {0.f, 0.f, 0.f, 0.f};
  for (int o0 = lo; o0 < o_end; o0 += q_tile) {
    const int nq = min(q_tile, o_end - o0);
    __syncthreads();
    if (tid < kRows) {
      const int hh = tid / q_tile, qi = tid % q_tile;
      if (tid < G * q_tile && qi < nq) {
        const int pos = text_idx[o0 + qi];
        const int h = g * G + hh;
        s_rows[tid] = q + static_cast<int64_t>(pos) * q_stride + static_cast<int64_t>(h) * d;
        s_rpos[tid] = pos;
        s_rlse[tid] = lse[static_cast<int64_t>(h) * lse_stride + pos] * lse_mul;
      } else {
        s_rows[tid] = nullptr;
        s_rpos[tid] = -1;
        s_rlse[tid] = 0.f;
      }
    }
    __syncthreads();
    load_rows_f32(Qs, s_rows, kRows, d);
    __syncthreads();
    float acc[4][4] = {};
    for (int e = 0; e < d; ++e) {
      float ka[4], qb[4];
#pragma unroll
      for (int a = 0; a < 4; ++a) ka[a] = Ks[(ty * 4 + a) * (d + 1) + e];
#pragma unroll
      for (int c = 0; c < 4; ++c) qb[c] = Qs[(tx + 16 * c) * (d + 1) + e];
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a][c] = fmaf(ka[a], qb[c], acc[a][c]);
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int row = tx + 16 * c;
      const int qpos = s_rpos[row];
      const float l2 = s_rlse[row];
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const int key = ty * 4 + a;
        if (qpos >= 0 && key < nk && qpos >= kp0 + key) mass[a] += exp2f(acc[a][c] * c2 - l2);
      }
    }
  }
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    float v = mass[a];
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int key = ty * 4 + a;
    if (tx == 0 && key < nk) partial[static_cast<int64_t>(g) * T + kp0 + key] = v;
  }
}

// ---------------------------------------------------------------- finalize
__global__ void __launch_bounds__(kThreads)
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

}  // namespace

int attn_q_tile(int Hq, int Hkv) {
  const int G = Hq / Hkv;
  const int qt = kRows / G;
  return qt > 0 ? qt : 1;
}

cudaError_t launch_score_attn(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                              int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s) {
  if (L.n_images == 0 || L.n_tokens == 0) return cudaSuccess;
  const int d = sa.head_dim, Hq = sa.n_q_heads, Hkv = sa.n_kv_heads;
  const int q_tile = attn_q_tile(Hq, Hkv);
  const float c2 = sa.softmax_scale * kLog2e;
  const size_t smem = static_cast<size_t>(kRows + kKT) * (d + 1) * sizeof(float);
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_lse, cudaFuncAttributeMaxDynamicSharedMemorySize, 80 * 1024);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_attn_mass, cudaFuncAttributeMaxDynamicSharedMemorySize, 80 * 1024);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const DevStatus* st = ws_at<DevStatus>(ws, p.status);
  const int32_t* text_idx = ws_at<int32_t>(ws, p.text_idx);
  const int32_t* text_cu = ws_at<int32_t>(ws, p.text_cu);
  const float* lse;
  int64_t lse_stride;
  float lse_mul;
  if (sa.lse == nullptr) {
    float* lse2 = ws_at<float>(ws, p.lse);
    const int64_t q_tiles = L.n_tokens / q_tile + L.n_requests;
    dim3 grid1(static_cast<unsigned>(q_tiles), static_cast<unsigned>(Hkv));
    cudaError_t e = launch_kernel(k_attn_lse, grid1, dim3(kThreads), smem, s, /*pdl=*/true,
                                  static_cast<const __nv_bfloat16*>(sa.q), sa.q_stride,
                                  static_cast<const __nv_bfloat16*>(sa.k), sa.k_stride, Hq, Hkv, d, c2, L.cu_seqlens,
                                  L.n_requests, text_idx, text_cu, ws_at<int32_t>(ws, p.qtile_cu), q_tile, lse2,
                                  L.n_tokens, st);
    if (e != cudaSuccess) return e;
    lse = lse2;
    lse_stride = L.n_tokens;
    lse_mul = 1.f;
  } else {
    lse = sa.lse;
    lse_stride = sa.lse_stride;
    lse_mul = kLog2e;  // natural-log LSE -> log2 domain
  }
  float* partial = ws_at<float>(ws, p.partial);
  const int64_t k_tiles = L.n_tokens / kKT + L.n_images;
  dim3 grid2(static_cast<unsigned>(k_tiles), static_cast<unsigned>(Hkv));
  cudaError_t e = launch_kernel(k_attn_mass, grid2, dim3(kThreads), smem, s, /*pdl=*/true,
                                static_cast<const __nv_bfloat16*>(sa.q), sa.q_stride,
                                static_cast<const __nv_bfloat16*>(sa.k), sa.k_stride, Hq, Hkv, d, c2, L.cu_seqlens,
                                L.img_start, L.img_len, ws_at<int32_t>(ws, p.img_req), L.n_images, text_idx, text_cu,
                                ws_at<int32_t>(ws, p.ktile_cu), q_tile, lse, lse_stride, lse_mul, partial,
                                L.n_tokens, st);
  if (e != cudaSuccess) return e;
  const int64_t want = (L.n_tokens + kThreads - 1) / kThreads;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  const int grid3 = static_cast<int>(want < cap ? want : cap);
  return launch_kernel(k_attn_finalize, dim3(grid3), dim3(kThreads), 0, s, /*pdl=*/true, partial, Hq, Hkv,
                       L.n_tokens, L.cu_seqlens, L.img_start, ws_at<int32_t>(ws, p.vis_cu),
                       ws_at<int32_t>(ws, p.img_req), text_cu, L.n_images, scores, img_sums, st);
}

}  // namespace avtp
