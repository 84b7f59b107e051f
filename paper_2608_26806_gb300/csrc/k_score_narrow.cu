// Criterion B on the CUDA cores, for query sets too narrow to fill a tensor-core tile:
// the request's last token alone (the output token whose attention FAST-V ranks visual
// tokens by, paper §4.1), or requests with few text tokens. Same quantity as the
// tensor-core path (k_score_attn.cu):
//   s_t = 1/(Hq*|Q_r|) * sum_h sum_{q in Q_r, pos q >= pos t} exp2(z2(h,q,t) - lse2(h,q)),
//   z2 = softmax_scale * log2(e) * q_h . k_{g(h)},  lse2 = log2 sum_{visible keys} exp2(z2).
//
// Rows: for KV group g, row o*G + j is query ordinal o with head g*G + j; the ordinal
// is the request index for the last-token set and the text ordinal for the text set.
//
// k_narrow_lse (pass 1): one CTA per (request, KV group, key split); a thread owns one
// key at a time (its d elements read as 16-byte vectors; the request's rows, in blocks
// of kRB, sit in shared memory as fp32) and keeps an online (max, sum) per row of the
// block; the CTA leaves one partial per (row, split).
// k_narrow_merge: merges the splits into lse2 per row (a warp per row), or converts a
// supplied natural-log LSE, and clears the per-key mass accumulator.
// k_narrow_mass (pass 2): one CTA per (key tile of an image, KV group), a thread per key:
// the key's probability under every row whose query follows it, summed and added to the
// 64-bit fixed-point accumulator that k_attn_finalize turns into scores.
// The work per key is d FMAs per row: memory-bound for a few rows, compute-bound beyond
// a few dozen, where the tensor-core path takes over (avtp_api.cu picks the path).
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kNT = 128;      // threads per CTA; pass 2 handles a 128-key tile
constexpr int kRB = 8;        // rows held in registers at a time
constexpr float kLog2e = 1.4426950408889634f;
constexpr unsigned long long kMassNotFinite = 1ull << 63;
static_assert(kNT == kAttnTileM, "pass 2 works on the key tiles of the tensor-core path");

struct NarrowArgs {
  const __nv_bfloat16* q;
  int64_t q_stride;
  const __nv_bfloat16* k;
  int64_t k_stride;
  const int32_t* cu;
  int R;
  const int32_t* text_idx;
  const int32_t* text_cu;
  const int32_t* ktile_cu;
  const int32_t* ktile_img;
  const int32_t* img_req;
  const int32_t* ist;
  const int32_t* iln;
  int NI;
  int Hq, Hkv, G, d;
  float c2;         // softmax_scale * log2(e)
  int last;         // 1: the request's last token is the only query
  int NS;           // key splits per (request, KV group) in pass 1
  int64_t rows;     // rows per KV group: queries of the batch (at most) times G
  float2* part;     // [Hkv][NS][rows]: pass-1 (max2, sum) per split
  float* lse2;      // [Hkv][rows]
  unsigned long long* mass;  // [key tiles][128], 2^-kAttnMassFracBits
  int64_t n_mass;
  const float* lse;          // supplied natural-log LSE [Hq][lse_stride], or null
  int64_t lse_stride;
  DevStatus* st;
};

// The request's first query ordinal and its number of queries.
__device__ __forceinline__ void request_queries(const NarrowArgs& a, int r, int64_t* o0, int* nq) {
  if (a.last) {
    *o0 = r;
    *nq = a.cu[r + 1] > a.cu[r] ? 1 : 0;
  } else {
    *o0 = a.text_cu[r];
    *nq = a.text_cu[r + 1] - a.text_cu[r];
  }
}

__device__ __forceinline__ int64_t query_pos(const NarrowArgs& a, int r, int64_t o) {
  return a.last ? static_cast<int64_t>(a.cu[r + 1]) - 1 : static_cast<int64_t>(a.text_idx[o]);
}

// (m, s) <- the online merge of (m, s) and (m2, s2), with -inf for "no key yet".
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  s = (m == -INFINITY ? 0.f : s * exp2f(m - M)) + (m2 == -INFINITY ? 0.f : s2 * exp2f(m2 - M));
  m = M;
}

// A block of up to kRB rows of request r, group g, starting at row rb: the queries as
// fp32 in shared memory, their positions, and (pass 2) their lse2.
struct RowBlock {
  float* qs;       // [kRB][d]
  int64_t* qpos;   // [kRB]; -1 for rows past the request's
  float* l2;       // [kRB]
};

__device__ void load_rows(const NarrowArgs& a, int r, int g, int64_t o0, int n_rows, int rb, const RowBlock& B,
                          bool want_lse) {
  const int d = a.d;
  for (int e = threadIdx.x; e < kRB * d / 8; e += kNT) {
    const int rr = e / (d / 8), c = e % (d / 8);
    const int row = rb + rr;
    float* dst = B.qs + rr * d + c * 8;
    if (row < n_rows) {
      const int64_t o = o0 + row / a.G;
      const int h = g * a.G + row % a.G;
      const int64_t pos = query_pos(a, r, o);
      const uint4 v = *reinterpret_cast<const uint4*>(a.q + pos * a.q_stride + static_cast<int64_t>(h) * d + c * 8);
      const uint32_t* w = reinterpret_cast<const uint32_t*>(&v);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        dst[2 * u] = __uint_as_float(w[u] << 16);
        dst[2 * u + 1] = __uint_as_float(w[u] & 0xffff0000u);
      }
    } else {
#pragma unroll
      for (int u = 0; u < 8; ++u) dst[u] = 0.f;
    }
  }
  for (int rr = threadIdx.x; rr < kRB; rr += kNT) {
    const int row = rb + rr;
    if (row < n_rows) {
      const int64_t o = o0 + row / a.G;
      B.qpos[rr] = query_pos(a, r, o);
      if (want_lse) B.l2[rr] = a.lse2[static_cast<int64_t>(g) * a.rows + o * a.G + row % a.G];
    } else {
      B.qpos[rr] = -1;
      if (want_lse) B.l2[rr] = 0.f;
    }
  }
}

// z[rr] = c2 * q_rr . k for the kRB rows of the block and key t of group g. All of the
// key's D/8 16-byte loads are issued before the first FMA: a key costs one memory round
// trip, not D/8 of them.
template <int D>
__device__ __forceinline__ void block_logits(const NarrowArgs& a, int64_t t, int g, const float* qs, float* z) {
  const uint4* kp = reinterpret_cast<const uint4*>(a.k + t * a.k_stride + static_cast<int64_t>(g) * D);
  uint4 kv[D / 8];
#pragma unroll
  for (int c = 0; c < D / 8; ++c) kv[c] = __ldg(kp + c);
  float acc[kRB];
#pragma unroll
  for (int rr = 0; rr < kRB; ++rr) acc[rr] = 0.f;
#pragma unroll
  for (int c = 0; c < D / 8; ++c) {
    const uint32_t* w = reinterpret_cast<const uint32_t*>(&kv[c]);
    float kf[8];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      kf[2 * u] = __uint_as_float(w[u] << 16);
      kf[2 * u + 1] = __uint_as_float(w[u] & 0xffff0000u);
    }
#pragma unroll
    for (int rr = 0; rr < kRB; ++rr) {
      const float4 q0 = *reinterpret_cast<const float4*>(qs + rr * D + c * 8);
      const float4 q1 = *reinterpret_cast<const float4*>(qs + rr * D + c * 8 + 4);
      float s = acc[rr];
      s = fmaf(kf[0], q0.x, s);
      s = fmaf(kf[1], q0.y, s);
      s = fmaf(kf[2], q0.z, s);
      s = fmaf(kf[3], q0.w, s);
      s = fmaf(kf[4], q1.x, s);
      s = fmaf(kf[5], q1.y, s);
      s = fmaf(kf[6], q1.z, s);
      s = fmaf(kf[7], q1.w, s);
      acc[rr] = s;
    }
  }
#pragma unroll
  for (int rr = 0; rr < kRB; ++rr) z[rr] = acc[rr] * a.c2;
}

// ---------------------------------------------------------------- pass 1
template <int D>
__global__ void __launch_bounds__(kNT)
k_narrow_lse(NarrowArgs a) {
  extern __shared__ __align__(16) float nsm[];
  __shared__ int64_t s_qpos[kRB];
  __shared__ float s_m[kNT / 32][kRB], s_s[kNT / 32][kRB];
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t units = static_cast<int64_t>(a.R) * a.Hkv * a.NS;
  for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
    const int sp = static_cast<int>(u % a.NS);
    const int g = static_cast<int>((u / a.NS) % a.Hkv);
    const int r = static_cast<int>(u / (static_cast<int64_t>(a.NS) * a.Hkv));
    int64_t o0;
    int nq;
    request_queries(a, r, &o0, &nq);
    const int n_rows = nq * a.G;
    if (n_rows == 0) continue;
    const int64_t t_lo = a.cu[r], T_r = a.cu[r + 1] - a.cu[r];
    const int64_t ks = t_lo + T_r * sp / a.NS, ke = t_lo + T_r * (sp + 1) / a.NS;
    for (int rb = 0; rb < n_rows; rb += kRB) {
      __syncthreads();  // the previous block's rows and reductions are no longer read
      const RowBlock B{nsm, s_qpos, nullptr};
      load_rows(a, r, g, o0, n_rows, rb, B, false);
      __syncthreads();
      float m[kRB], s[kRB];
#pragma unroll
      for (int rr = 0; rr < kRB; ++rr) { m[rr] = -INFINITY; s[rr] = 0.f; }
      for (int64_t t = ks + threadIdx.x; t < ke; t += kNT) {
        float z[kRB];
        block_logits<D>(a, t, g, nsm, z);
#pragma unroll
        for (int rr = 0; rr < kRB; ++rr) {
          if (t > s_qpos[rr]) continue;  // after the query (or a row past the request's)
          if (z[rr] > m[rr]) {
            s[rr] = (m[rr] == -INFINITY ? 0.f : s[rr] * exp2f(m[rr] - z[rr])) + 1.f;
            m[rr] = z[rr];
          } else {
            s[rr] += exp2f(z[rr] - m[rr]);
          }
        }
      }
      // reduce over the CTA: warps by shuffles, then across the warps
#pragma unroll
      for (int rr = 0; rr < kRB; ++rr) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, m[rr], off);
          const float s2 = __shfl_xor_sync(0xffffffffu, s[rr], off);
          merge_ms(m[rr], s[rr], m2, s2);
        }
        if (lane == 0) {
          s_m[warp][rr] = m[rr];
          s_s[warp][rr] = s[rr];
        }
      }
      __syncthreads();
      if (threadIdx.x < kRB && rb + static_cast<int>(threadIdx.x) < n_rows) {
        const int rr = threadIdx.x;
        float M = s_m[0][rr], Sm = s_s[0][rr];
        for (int w = 1; w < kNT / 32; ++w) merge_ms(M, Sm, s_m[w][rr], s_s[w][rr]);
        const int row = rb + rr;
        const int64_t ro = (o0 + row / a.G) * a.G + row % a.G;
        a.part[(static_cast<int64_t>(g) * a.NS + sp) * a.rows + ro] = make_float2(M, Sm);
      }
    }
  }
}

// ---------------------------------------------------------------- merge
__global__ void __launch_bounds__(256)
k_narrow_merge(NarrowArgs a, int64_t n_rows_used) {
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t tid0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  for (int64_t u = tid0; u < a.n_mass; u += stride) a.mass[u] = 0ull;
  // rows in use: R * G (last-token set) or (text tokens of the batch) * G
  const int64_t n_text = a.last ? 0 : a.text_cu[a.R];
  // a warp per row: the lanes merge the splits, then a shuffle tree
  const int lane = threadIdx.x & 31;
  const int64_t wstride = stride >> 5;
  for (int64_t u = tid0 >> 5; u < static_cast<int64_t>(a.Hkv) * n_rows_used; u += wstride) {
    const int g = static_cast<int>(u / n_rows_used);
    const int64_t ro = u % n_rows_used;
    const int64_t o = ro / a.G;
    if (!a.last && o >= n_text) continue;                        // no such text token in this batch
    if (a.last && a.cu[o + 1] == a.cu[o]) continue;              // a request without tokens has no query
    float l2;
    if (a.lse != nullptr) {
      const int h = g * a.G + static_cast<int>(ro % a.G);
      const int r = a.last ? static_cast<int>(o) : upper_index(a.text_cu, a.R, o);
      l2 = a.lse[static_cast<int64_t>(h) * a.lse_stride + query_pos(a, r, o)] * kLog2e;
    } else {
      float M = -INFINITY, Sm = 0.f;
      for (int sp = lane; sp < a.NS; sp += 32) {
        const float2 p = a.part[(static_cast<int64_t>(g) * a.NS + sp) * a.rows + ro];
        merge_ms(M, Sm, p.x, p.y);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, M, off);
        const float s2 = __shfl_xor_sync(0xffffffffu, Sm, off);
        merge_ms(M, Sm, m2, s2);
      }
      l2 = M + log2f(Sm);
    }
    if (lane == 0) a.lse2[static_cast<int64_t>(g) * a.rows + ro] = l2;
  }
}

// ---------------------------------------------------------------- pass 2
template <int D>
__global__ void __launch_bounds__(kNT)
k_narrow_mass(NarrowArgs a) {
  extern __shared__ __align__(16) float nsm[];
  __shared__ int64_t s_qpos[kRB];
  __shared__ float s_l2[kRB];
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int n_tiles = a.ktile_cu[a.NI];
  const int64_t units = static_cast<int64_t>(n_tiles) * a.Hkv;
  for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
    const int g = static_cast<int>(u % a.Hkv);
    const int tile = static_cast<int>(u / a.Hkv);
    const int i = a.ktile_img[tile];
    const int r = a.img_req[i];
    int64_t o0;
    int nq;
    request_queries(a, r, &o0, &nq);
    const int n_rows = nq * a.G;
    const int ok = (tile - a.ktile_cu[i]) * kNT + static_cast<int>(threadIdx.x);  // key within the image
    const bool has = ok < a.iln[i];
    const int64_t t = static_cast<int64_t>(a.cu[r]) + a.ist[i] + ok;
    float mass = 0.f;
    for (int rb = 0; rb < n_rows; rb += kRB) {
      __syncthreads();
      const RowBlock B{nsm, s_qpos, s_l2};
      load_rows(a, r, g, o0, n_rows, rb, B, true);
      __syncthreads();
      if (!has) continue;
      float z[kRB];
      block_logits<D>(a, t, g, nsm, z);
#pragma unroll
      for (int rr = 0; rr < kRB; ++rr)
        if (t <= s_qpos[rr]) mass += exp2f(z[rr] - s_l2[rr]);
    }
    if (has && n_rows > 0) {
      unsigned long long* dst = a.mass + static_cast<int64_t>(tile) * kNT + threadIdx.x;
      if (mass <= 512.f) {  // at most one per row
        atomicAdd(dst, static_cast<unsigned long long>(__float2ll_rn(mass * static_cast<float>(1ull << kAttnMassFracBits))));
      } else {
        atomicOr(dst, kMassNotFinite);  // NaN or inf inputs: the key scores NaN
      }
    }
  }
}

int narrow_splits(const avtp_layout_t& L, int Hkv) {
  const int64_t want = 4ll * device_sm_count();
  const int64_t per = static_cast<int64_t>(L.n_requests) * Hkv;
  int64_t ns = (want + per - 1) / per;
  return static_cast<int>(ns < 1 ? 1 : (ns > kNarrowMaxSplits ? kNarrowMaxSplits : ns));
}

}  // namespace

NarrowPlan narrow_plan(const avtp_layout_t& L, const avtp_score_args_t& sa, int64_t max_text) {
  NarrowPlan p;
  p.G = sa.n_q_heads / sa.n_kv_heads;
  p.rows = (sa.query_set == AVTP_QUERIES_LAST ? static_cast<int64_t>(L.n_requests) : max_text) * p.G;
  p.NS = narrow_splits(L, sa.n_kv_heads);
  return p;
}

cudaError_t launch_score_narrow(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores, int64_t* img_sums,
                                void* ws, const WsPlan& p, const AttnPlan& plan, cudaStream_t s) {
  if (L.n_images == 0 || L.n_tokens == 0) return cudaSuccess;
  const NarrowPlan np = narrow_plan(L, sa, plan.max_text);
  NarrowArgs a{};
  a.q = static_cast<const __nv_bfloat16*>(sa.q);
  a.q_stride = sa.q_stride;
  a.k = static_cast<const __nv_bfloat16*>(sa.k);
  a.k_stride = sa.k_stride;
  a.cu = L.cu_seqlens;
  a.R = L.n_requests;
  a.text_idx = ws_at<int32_t>(ws, p.text_idx);
  a.text_cu = ws_at<int32_t>(ws, p.text_cu);
  a.ktile_cu = ws_at<int32_t>(ws, p.ktile_cu);
  a.ktile_img = ws_at<int32_t>(ws, p.ktile_img);
  a.img_req = ws_at<int32_t>(ws, p.img_req);
  a.ist = L.img_start;
  a.iln = L.img_len;
  a.NI = L.n_images;
  a.Hq = sa.n_q_heads;
  a.Hkv = sa.n_kv_heads;
  a.G = np.G;
  a.d = sa.head_dim;
  a.c2 = sa.softmax_scale * kLog2e;
  a.last = sa.query_set == AVTP_QUERIES_LAST ? 1 : 0;
  a.NS = np.NS;
  a.rows = np.rows;
  a.part = ws_at<float2>(ws, p.p1_part);
  a.lse2 = ws_at<float>(ws, p.lse_rows);
  a.mass = ws_at<unsigned long long>(ws, p.mass);
  a.n_mass = plan.n_ktiles_max * kAttnTileM;
  a.lse = sa.lse;
  a.lse_stride = sa.lse_stride;
  a.st = ws_at<DevStatus>(ws, p.status);
  const size_t qsm = static_cast<size_t>(kRB) * sa.head_dim * sizeof(float);
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  if (sa.lse == nullptr) {
    const int64_t units = static_cast<int64_t>(L.n_requests) * a.Hkv * a.NS;
    const int grid = static_cast<int>(units < cap ? units : cap);
    cudaError_t e = sa.head_dim == 64 ? launch_kernel(k_narrow_lse<64>, dim3(grid), dim3(kNT), qsm, s, true, a)
                                      : launch_kernel(k_narrow_lse<128>, dim3(grid), dim3(kNT), qsm, s, true, a);
    if (e != cudaSuccess) return e;
  }
  {
    const int64_t work = (a.n_mass > 32 * a.Hkv * a.rows ? a.n_mass : 32 * a.Hkv * a.rows);
    const int64_t want = (work + 255) / 256;
    const int grid = static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
    cudaError_t e = launch_kernel(k_narrow_merge, dim3(grid), dim3(256), 0, s, /*pdl=*/true, a, a.rows);
    if (e != cudaSuccess) return e;
  }
  const int64_t units2 = plan.n_ktiles_max * a.Hkv;
  const int grid2 = static_cast<int>(units2 < 1 ? 1 : (units2 < cap ? units2 : cap));
  cudaError_t e = sa.head_dim == 64 ? launch_kernel(k_narrow_mass<64>, dim3(grid2), dim3(kNT), qsm, s, true, a)
                                    : launch_kernel(k_narrow_mass<128>, dim3(grid2), dim3(kNT), qsm, s, true, a);
  if (e != cudaSuccess) return e;
  return launch_attn_finalize(L, sa, scores, img_sums, ws, p, plan, s);
}

}  // namespace avtp
