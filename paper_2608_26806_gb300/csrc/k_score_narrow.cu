// Criterion B on the CUDA cores, for query sets too narrow to fill a tensor-core tile:
// the request's last token alone (the output token whose attention FAST-V ranks visual
// tokens by, paper §4.1), or requests with few text tokens. Same quantity as the
// tensor-core path (k_score_attn.cu):
//   s_t = 1/(Hq*|Q_r|) * sum_h sum_{q in Q_r, pos q >= pos t} exp2(z2(h,q,t) - lse2(h,q)),
//   z2 = softmax_scale * log2(e) * q_h . k_{g(h)},  lse2 = log2 sum_{visible keys} exp2(z2).
//
// Rows: the global row of query ordinal o and head h is o*Hq + h; the ordinal is the
// request index for the last-token set and the text ordinal for the text set.
//
// The keys are read once. k_narrow_logits: one CTA per (request, KV group, key split);
// each warp takes 16-key tiles and multiplies them by the group's rows, 8 at a time, with
// warp-level mma.sync (m16n8k16, bf16 in, fp32 accumulate): a tile too narrow for a
// tcgen05 MMA still gets the tensor cores, and all of a tile's key loads are in flight
// before its first MMA. (Holding the rows in shared memory and a key per thread with
// fp32 FMAs spent 29 % of its issue slots on shared-memory loads and ran 24 us for the
// 20 MB of keys of a 9856-token request.) It
// writes every logit z2 of the request's rows to a buffer (rows x keys of the request,
// fp32: 1.3 MB for one query token over 9856 keys and 32 heads) and, unless the LSE is
// supplied, one online (max, sum) partial per (row, split). k_narrow_mass: each CTA
// merges the partials of its request's rows into lse2 (one round of loads), then a thread
// per visual key sums exp2(z2 - lse2) over the rows whose query follows it, reading the
// logits back (coalesced: consecutive keys of a row are consecutive), and writes the key's
// score, formed from the fixed-point mass as k_attn_finalize forms it, and the tile's share
// of its image's fixed-point sum (one atomic per tile). No key is read twice, and no
// finalising kernel follows.
// The work per key is d multiply-adds per row; the logits buffer grows with the rows, and
// for wide query sets the tcgen05 path takes over (avtp_api.cu picks the path).
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kNT = 128;      // threads per CTA; k_narrow_mass handles a 128-key tile
constexpr int kRB = 8;        // rows per MMA tile (the N of m16n8k16)
constexpr int kMassRows = 256;  // rows whose lse2 and query position k_narrow_mass stages at a time
constexpr int kMassBatch = 32;  // logits a thread of k_narrow_mass loads at once
constexpr int kSplitLanes = 4;  // lanes that merge one row's split partials in k_narrow_mass
static_assert(kNarrowMaxSplits % kSplitLanes == 0 && 32 % kSplitLanes == 0, "split lanes");
constexpr float kLog2e = 1.4426950408889634f;
static_assert(kNT == kAttnTileM, "k_narrow_mass works on the key tiles of the tensor-core path");

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
  int NS;           // key splits per (request, KV group) in k_narrow_logits
  float* z;         // logits, request by request: [rows of r][T_r]
  float2* part;     // [global rows][NS]: (max2, sum) per split
  float* scores;             // [T]: the visual keys' scores
  int64_t* img_sums;         // [n_img]: fixed-point image sums (zeroed by the validation kernel)
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

// Offset of request r's logits: Hq * sum over earlier requests of queries x tokens.
__device__ __forceinline__ int64_t logits_base(const NarrowArgs& a, int r) {
  if (a.last) return static_cast<int64_t>(a.Hq) * a.cu[r];
  int64_t s = 0;
  for (int u = 0; u < r; ++u)
    s += static_cast<int64_t>(a.text_cu[u + 1] - a.text_cu[u]) * (a.cu[u + 1] - a.cu[u]);
  return s * a.Hq;
}

// (m, s) <- the online merge of (m, s) and (m2, s2), with -inf for "no key yet".
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  s = (m == -INFINITY ? 0.f : s * exp2f(m - M)) + (m2 == -INFINITY ? 0.f : s2 * exp2f(m2 - M));
  m = M;
}

// ---------------------------------------------------------------- the logits (and lse2)
// D = q . k for a 16-key x 8-row tile on the tensor cores (mma.sync m16n8k16, bf16 in,
// fp32 accumulate): the keys are the 16-row A operand, the 8 rows of a block the B
// operand. Lane l holds keys l/4 and l/4 + 8 of the tile and rows 2(l%4), 2(l%4) + 1.
__device__ __forceinline__ void mma_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <int D>
__global__ void __launch_bounds__(kNT)
k_narrow_logits(NarrowArgs a) {
  constexpr int KS = D / 16;  // k-steps
  __shared__ float s_m[kNT / 32][kRB], s_s[kNT / 32][kRB];
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int kq = 2 * (lane & 3);  // this lane's column pair in a k-step
  const int km = lane >> 2;       // this lane's keys in a tile: km and km + 8
  const bool want_lse = a.lse == nullptr;
  const int64_t units = static_cast<int64_t>(a.R) * a.Hkv * a.NS;
  for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
    const int sp = static_cast<int>(u % a.NS);
    const int g = static_cast<int>((u / a.NS) % a.Hkv);
    const int r = static_cast<int>(u / (static_cast<int64_t>(a.NS) * a.Hkv));
    int64_t o0;
    int nq;
    request_queries(a, r, &o0, &nq);
    const int n_rows = nq * a.G;
    const int64_t t_lo = a.cu[r], T_r = a.cu[r + 1] - a.cu[r];
    const int64_t ks = t_lo + T_r * sp / a.NS, ke = t_lo + T_r * (sp + 1) / a.NS;
    const int64_t zb = logits_base(a, r);
    for (int rb = 0; rb < n_rows; rb += kRB) {
      // B operand: row rb + km of the block (the lane's row for the loads), as bf16 pairs
      uint32_t bq[KS][2];
      {
        const int row = rb + km;
        if (row < n_rows) {
          const int64_t o = o0 + row / a.G;
          const int h = g * a.G + row % a.G;
          const __nv_bfloat16* qp = a.q + query_pos(a, r, o) * a.q_stride + static_cast<int64_t>(h) * D;
#pragma unroll
          for (int kk = 0; kk < KS; ++kk) {
            bq[kk][0] = *reinterpret_cast<const uint32_t*>(qp + kk * 16 + kq);
            bq[kk][1] = *reinterpret_cast<const uint32_t*>(qp + kk * 16 + 8 + kq);
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < KS; ++kk) bq[kk][0] = bq[kk][1] = 0u;
        }
      }
      // the lane's two rows of the C tile: where their logits go, their query positions
      int64_t zrow[2], qp[2];
      bool live[2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int row = rb + kq + j;
        live[j] = row < n_rows;
        const int64_t o_loc = row / a.G, h = g * a.G + row % a.G;
        zrow[j] = zb + (o_loc * a.Hq + h) * T_r - t_lo;
        qp[j] = live[j] ? query_pos(a, r, o0 + o_loc) : -1;
      }
      float m[2] = {-INFINITY, -INFINITY}, sm[2] = {0.f, 0.f};
      // two tiles per step: every A load of both in flight before the first MMA
      for (int64_t t0 = ks + warp * 32; t0 < ke; t0 += (kNT / 32) * 32) {
        uint32_t ak[2][KS][4];
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int64_t tA = t0 + 16 * h2 + km, tB = tA + 8;
          const __nv_bfloat16* kA = a.k + tA * a.k_stride + static_cast<int64_t>(g) * D;
          const __nv_bfloat16* kB = a.k + tB * a.k_stride + static_cast<int64_t>(g) * D;
#pragma unroll
          for (int kk = 0; kk < KS; ++kk) {
            ak[h2][kk][0] = tA < ke ? __ldg(reinterpret_cast<const unsigned int*>(kA + kk * 16 + kq)) : 0u;
            ak[h2][kk][1] = tB < ke ? __ldg(reinterpret_cast<const unsigned int*>(kB + kk * 16 + kq)) : 0u;
            ak[h2][kk][2] = tA < ke ? __ldg(reinterpret_cast<const unsigned int*>(kA + kk * 16 + 8 + kq)) : 0u;
            ak[h2][kk][3] = tB < ke ? __ldg(reinterpret_cast<const unsigned int*>(kB + kk * 16 + 8 + kq)) : 0u;
          }
        }
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int64_t tA = t0 + 16 * h2 + km, tB = tA + 8;
          float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int kk = 0; kk < KS; ++kk)
            mma_16816(c, ak[h2][kk][0], ak[h2][kk][1], ak[h2][kk][2], ak[h2][kk][3], bq[kk][0], bq[kk][1]);
          // c[0], c[1]: key tA, rows kq, kq + 1; c[2], c[3]: key tB, the same rows
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int j = e & 1;
            const int64_t t = e < 2 ? tA : tB;
            if (!live[j] || t >= ke) continue;
            const float z = c[e] * a.c2;
            a.z[zrow[j] + t] = z;
            if (!want_lse || t > qp[j]) continue;  // the key follows the query
            if (z > m[j]) {
              sm[j] = (m[j] == -INFINITY ? 0.f : sm[j] * exp2f(m[j] - z)) + 1.f;
              m[j] = z;
            } else {
              sm[j] += exp2f(z - m[j]);
            }
          }
        }
      }
      if (!want_lse) continue;
      // reduce over the lanes that hold the same rows (same l % 4), then over the warps
#pragma unroll
      for (int j = 0; j < 2; ++j) {
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, m[j], off);
          const float s2 = __shfl_xor_sync(0xffffffffu, sm[j], off);
          merge_ms(m[j], sm[j], m2, s2);
        }
      }
      __syncthreads();  // s_m / s_s of the previous block are no longer read
      if (lane < 4) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          s_m[warp][kq + j] = m[j];
          s_s[warp][kq + j] = sm[j];
        }
      }
      __syncthreads();
      if (threadIdx.x < kRB && rb + static_cast<int>(threadIdx.x) < n_rows) {
        const int rr = threadIdx.x;
        float M = s_m[0][rr], Sm = s_s[0][rr];
        for (int w = 1; w < kNT / 32; ++w) merge_ms(M, Sm, s_m[w][rr], s_s[w][rr]);
        const int row = rb + rr;
        const int64_t gr = (o0 + row / a.G) * a.Hq + g * a.G + row % a.G;
        a.part[gr * a.NS + sp] = make_float2(M, Sm);
      }
    }
  }
}

// ---------------------------------------------------------------- the mass of every visual key
__global__ void __launch_bounds__(kNT)
k_narrow_mass(NarrowArgs a) {
  __shared__ float s_l2[kMassRows];
  __shared__ int64_t s_qpos[kMassRows];
  __shared__ long long s_fx[kNT / 32];
  pdl_wait();
  pdl_trigger();
  if (!a.st->layout_ok) return;
  const int n_tiles = a.ktile_cu[a.NI];
  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int i = a.ktile_img[tile];
    const int r = a.img_req[i];
    int64_t o0;
    int nq;
    request_queries(a, r, &o0, &nq);
    const int64_t n_rows = static_cast<int64_t>(nq) * a.Hq;
    const int ok = (tile - a.ktile_cu[i]) * kNT + static_cast<int>(threadIdx.x);  // key within the image
    const bool has = ok < a.iln[i];
    const int64_t t_lo = a.cu[r], T_r = a.cu[r + 1] - a.cu[r];
    const int64_t t = t_lo + a.ist[i] + ok;
    const float* zr = a.z + logits_base(a, r) + (t - t_lo);
    float mass = 0.f;
    for (int64_t rb = 0; rb < n_rows; rb += kMassRows) {
      const int nr = static_cast<int>(n_rows - rb < kMassRows ? n_rows - rb : kMassRows);
      // the first kMassBatch logits of the key, loaded while the rows are staged
      float zz0[kMassBatch];
#pragma unroll
      for (int j = 0; j < kMassBatch; ++j) zz0[j] = has && j < nr ? __ldcg(zr + (rb + j) * T_r) : 0.f;
      __syncthreads();
      for (int rr = threadIdx.x; rr < kMassRows; rr += kNT) {
        const int64_t row = rb + rr;
        if (row < n_rows) {
          const int64_t o = o0 + row / a.Hq;
          const int h = static_cast<int>(row % a.Hq);
          const int64_t pos = query_pos(a, r, o);
          s_qpos[rr] = pos;
          if (a.lse != nullptr) s_l2[rr] = a.lse[static_cast<int64_t>(h) * a.lse_stride + pos] * kLog2e;
        } else {
          s_qpos[rr] = -1;
          s_l2[rr] = 0.f;
        }
      }
      if (a.lse == nullptr) {
        // lse2 of the staged rows from the logits pass's (max, sum) partials: kSplitLanes
        // lanes per row, every partial load of a lane issued before it merges
        const int sub = threadIdx.x % kSplitLanes;
        for (int rr0 = static_cast<int>(threadIdx.x) / kSplitLanes; rr0 < kMassRows; rr0 += kNT / kSplitLanes) {
          float M = -INFINITY, Sm = 0.f;
          if (rr0 < nr) {
            const float2* pp = a.part + ((o0 * a.Hq) + rb + rr0) * a.NS;
            float2 pv[kNarrowMaxSplits / kSplitLanes];
#pragma unroll
            for (int q = 0; q < kNarrowMaxSplits / kSplitLanes; ++q) {
              const int sp = sub + q * kSplitLanes;
              pv[q] = sp < a.NS ? __ldcg(pp + sp) : make_float2(-INFINITY, 0.f);
            }
#pragma unroll
            for (int q = 0; q < kNarrowMaxSplits / kSplitLanes; ++q) merge_ms(M, Sm, pv[q].x, pv[q].y);
          }
#pragma unroll
          for (int off = kSplitLanes / 2; off > 0; off >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, M, off);
            const float s2 = __shfl_xor_sync(0xffffffffu, Sm, off);
            merge_ms(M, Sm, m2, s2);
          }
          if (sub == 0 && rr0 < nr) s_l2[rr0] = M + log2f(Sm);
        }
      }
      __syncthreads();
      if (!has) continue;
#pragma unroll
      for (int j = 0; j < kMassBatch; ++j)
        if (j < nr && t <= s_qpos[j]) mass += exp2f(zz0[j] - s_l2[j]);
      // the rest, kMassBatch logits in flight before the first exp2
      for (int r0 = kMassBatch; r0 < nr; r0 += kMassBatch) {
        float zz[kMassBatch];
#pragma unroll
        for (int j = 0; j < kMassBatch; ++j) zz[j] = r0 + j < nr ? __ldcg(zr + (rb + r0 + j) * T_r) : 0.f;
#pragma unroll
        for (int j = 0; j < kMassBatch; ++j)
          if (r0 + j < nr && t <= s_qpos[r0 + j]) mass += exp2f(zz[j] - s_l2[r0 + j]);
      }
    }
    // the score, as k_attn_finalize forms it from the fixed-point mass: s = mass * 2^-40 /
    // (Hq * |Q_r|), NaN for a mass that is not a finite number (non-finite inputs)
    long long fx = 0;
    if (has) {
      float sc = 0.f;
      if (n_rows > 0) {
        if (mass <= 4194304.f) {
          const long long m = __float2ll_rn(mass * static_cast<float>(1ull << kAttnMassFracBits));
          sc = __ll2float_rn(m) * (1.0f / static_cast<float>(1ull << kAttnMassFracBits));
          sc = sc / static_cast<float>(n_rows);
        } else {
          sc = __int_as_float(0x7fc00000);
        }
      }
      a.scores[t] = sc;
      fx = fixed_point_score(sc);
    }
    // the tile's share of its image's fixed-point sum, one atomic
    fx = warp_sum(fx);
    if ((threadIdx.x & 31) == 0) s_fx[threadIdx.x >> 5] = fx;
    __syncthreads();
    if (threadIdx.x == 0) {
      long long sum = 0;
#pragma unroll
      for (int w = 0; w < kNT / 32; ++w) sum += s_fx[w];
      atomicAdd(reinterpret_cast<unsigned long long*>(a.img_sums + i), static_cast<unsigned long long>(sum));
    }
    __syncthreads();  // s_fx is read before the next tile writes it
  }
}

// Key splits per (request, KV group): about two keys per thread of a unit, on average
// over the requests.
int narrow_splits(const avtp_layout_t& L, int Hkv) {
  (void)Hkv;
  const int64_t per_request = L.n_tokens / (L.n_requests > 0 ? L.n_requests : 1);
  const int64_t ns = (per_request + 2 * kNT - 1) / (2 * kNT);
  return static_cast<int>(ns < 1 ? 1 : (ns > kNarrowMaxSplits ? kNarrowMaxSplits : ns));
}

}  // namespace

NarrowPlan narrow_plan(const avtp_layout_t& L, const avtp_score_args_t& sa, int64_t max_text) {
  NarrowPlan p;
  p.G = sa.n_q_heads / sa.n_kv_heads;
  const int64_t n_q = sa.query_set == AVTP_QUERIES_LAST ? static_cast<int64_t>(L.n_requests) : max_text;
  p.rows = n_q * sa.n_q_heads;
  p.NS = narrow_splits(L, sa.n_kv_heads);
  // logits: Hq x queries x tokens of each request, at most Hq x n_q x T (the last-token set:
  // Hq x T exactly)
  p.z_elems = sa.query_set == AVTP_QUERIES_LAST ? static_cast<int64_t>(sa.n_q_heads) * L.n_tokens
                                                : (n_q > 0 && L.n_tokens > INT64_MAX / 4 / n_q / sa.n_q_heads
                                                       ? INT64_MAX / 4
                                                       : p.rows * L.n_tokens);
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
  a.z = ws_at<float>(ws, p.zbuf);
  a.part = ws_at<float2>(ws, p.p1_part);
  a.st = ws_at<DevStatus>(ws, p.status);
  a.scores = scores;
  a.img_sums = img_sums;
  a.lse = sa.lse;
  a.lse_stride = sa.lse_stride;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  const int64_t units = static_cast<int64_t>(L.n_requests) * a.Hkv * a.NS;
  const int grid = static_cast<int>(units < cap ? units : cap);
  cudaError_t e = sa.head_dim == 64 ? launch_kernel(k_narrow_logits<64>, dim3(grid), dim3(kNT), 0, s, true, a)
                                    : launch_kernel(k_narrow_logits<128>, dim3(grid), dim3(kNT), 0, s, true, a);
  if (e != cudaSuccess) return e;
  const int64_t units2 = plan.n_ktiles_max;
  const int grid2 = static_cast<int>(units2 < 1 ? 1 : (units2 < cap ? units2 : cap));
  return launch_kernel(k_narrow_mass, dim3(grid2), dim3(kNT), 0, s, true, a);
}

}  // namespace avtp
