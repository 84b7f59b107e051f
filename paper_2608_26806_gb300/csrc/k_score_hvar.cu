// Criterion A (paper §3.3.1): I_v = 1 - cos(h^l_v, h^prior_v) for every visual token.
//
// HBM-bound stream: each visual row of h_cur and h_prior is read once (2 x D x 2
// bytes per token). Rows are staged through shared memory by bulk asynchronous
// copies (cp.async.bulk, completion on an mbarrier): every warp runs its own
// 3-deep pipeline of row chunks (2 x 2 KiB), so about 12 KiB per warp and
// 192 KiB per SM are in flight, independent of the register file. The warp then
// accumulates dot, |a|^2 and |b|^2 in fp32 from shared memory.
//
// Work is split by visual ordinal, whole tokens per warp: each warp first takes a
// fixed contiguous run of about 80 % of its even share, then draws the remaining
// tokens one at a time from a pool (a counter in the status word that the validation
// kernel resets; the first draw waits for that kernel). Without the pool the CTAs
// finished up to 6 us apart on the Qwen3-VL-8B-shaped request: SMs do not all get the
// same share of the memory bandwidth. A token is scored by one warp either way, so the
// scores do not depend on which warp takes it. Each CTA derives the ordinal -> (image,
// packed position) map itself from the layout, staged in shared memory, so it needs
// nothing from the validation kernel before its pool draws and runs alongside it
// (programmatic dependent launch). Every position is checked to lie in [0, T) before a
// copy is issued, so a malformed layout cannot make it read out of bounds; the
// validation kernel reports it. Layouts too large to stage fall back to the validation
// kernel's prefix arrays.
//
// Per-image sums S_i = sum rint(fx(I) * 2^32) (integers, so any order gives the
// same value) are accumulated per warp over runs of rows of the same image and
// added to img_sums with one atomic per run. The validation kernel zeroes
// img_sums, so the first atomic of a warp waits for it; that is normally well after
// it has finished.
//
// L2 policy: h_prior evict-first, h_cur evict-last, because the compaction step
// reads the kept h_cur rows again right after.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kWarps = 16;                // warps per CTA, each with its own pipeline
constexpr int kThreads = kWarps * 32;
constexpr int kSlots = 3;                 // pipeline depth per warp
constexpr int kChunkElems = 1024;         // bf16 per tensor per slot (2 KiB)
constexpr int kChunkBytes = kChunkElems * 2;
constexpr int kSlotBytes = 2 * kChunkBytes;
constexpr size_t kSmemBytes = static_cast<size_t>(kWarps) * kSlots * kSlotBytes;  // 192 KiB
// Layouts up to this many images / requests are staged in shared memory (about 11 KiB
// with the barriers, next to the 192-KiB pipeline).
constexpr int kStageImages = 1024;
constexpr int kStageRequests = 256;

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(smem_addr(bar)),
      "r"(bytes)
      : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::
          "r"(smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

// Two fp32 FMAs in one instruction (fma.rn.f32x2), each rounded as fmaf would be.
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

// Ordinal -> packed position map: image i covers visual ordinals [vcu[i], vcu[i+1])
// and starts at packed position gstart[i].
struct VisMap {
  const int32_t* vcu;     // [NI + 1]
  const int32_t* gstart;  // [NI] (staged) or nullptr (then cu[req[i]] + ist[i])
  const int32_t* req;     // [NI] (unstaged path)
  const int32_t* cu;
  const int32_t* ist;
  int NI;
  int64_t n_vis;
  __device__ int64_t position(int64_t v, int& img) const {
    if (!(vcu[img] <= v && v < vcu[img + 1])) img = upper_index(vcu, NI, v);
    const int64_t start = gstart ? gstart[img] : static_cast<int64_t>(cu[req[img]]) + ist[img];
    return start + (v - vcu[img]);
  }
};

// Exclusive scan over n values of a shared array, in place, by the whole block; out[n] = total.
__device__ void block_scan_inplace(int32_t* a, int n, int32_t* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int per = (n + kThreads - 1) / kThreads;
  const int b0 = threadIdx.x * per, b1 = min(n, b0 + per);
  int32_t sum = 0;
  for (int j = b0; j < b1; ++j) sum += a[j];
  int32_t x = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  int32_t pre = 0, tot = 0;
  for (int w = 0; w < kWarps; ++w) {
    pre += (w < warp) ? s_warp[w] : 0;
    tot += s_warp[w];
  }
  int32_t run = pre + x - sum;
  __syncthreads();
  for (int j = b0; j < b1; ++j) {
    const int32_t v = a[j];
    a[j] = run;
    run += v;
  }
  if (threadIdx.x == 0) a[n] = tot;
  __syncthreads();
}

// 64 registers a thread: on large batches (no SMs left free) a CTA of the selection
// kernel (256 threads, up to 128 registers) can then start on the same SM as this one
// and wait there for the scores.
__global__ void __maxnreg__(64)
k_score_hvar(const __nv_bfloat16* __restrict__ h_cur, int64_t cur_stride, const __nv_bfloat16* __restrict__ h_prior,
             int64_t prior_stride, int D, const int32_t* __restrict__ cu, int R, const int32_t* __restrict__ icu,
             const int32_t* __restrict__ ist, const int32_t* __restrict__ iln, int NI, int64_t T,
             const int32_t* __restrict__ prep_vis_cu, const int32_t* __restrict__ prep_img_req,
             float* __restrict__ scores, int64_t* __restrict__ img_sums, DevStatus* st) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ uint64_t bars[kWarps][kSlots];
  __shared__ int32_t s_vcu[kStageImages + 1];
  __shared__ int32_t s_gstart[kStageImages];
  __shared__ int32_t s_icu[kStageRequests + 1];
  __shared__ int32_t s_cu[kStageRequests + 1];
  __shared__ int32_t s_warp[kWarps];
  pdl_trigger();
#ifdef AVTP_TIMELINE
  __shared__ unsigned s_tl_done;
  if (threadIdx.x == 0) {
    s_tl_done = 0;
    timeline_stamp(st, kTlScoreBegin);
  }
  __syncthreads();
#endif
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  unsigned char* wbuf = smem + static_cast<size_t>(warp) * kSlots * kSlotBytes;
  uint64_t* wbar = bars[warp];
  if (lane == 0) {
    for (int s = 0; s < kSlots; ++s) mbar_init(&wbar[s], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }

  // ---- ordinal map
  VisMap map;
  map.cu = cu;
  map.ist = ist;
  map.NI = NI;
  const bool staged = NI <= kStageImages && R <= kStageRequests;
  if (staged) {
    // all four layout arrays in one round of loads, so that one DRAM latency (not two)
    // precedes the first bulk copy
    for (int j = threadIdx.x; j <= R; j += kThreads) {
      s_icu[j] = min(max(icu[j], 0), NI);
      s_cu[j] = cu[j];
    }
    for (int j = threadIdx.x; j < NI; j += kThreads) {
      s_vcu[j] = max(iln[j], 0);
      s_gstart[j] = ist[j];
    }
    __syncthreads();
    block_scan_inplace(s_vcu, NI, s_warp);
    for (int j = threadIdx.x; j < NI; j += kThreads) s_gstart[j] += s_cu[upper_index(s_icu, R, j)];  // request of j
    __syncthreads();
    map.vcu = s_vcu;
    map.gstart = s_gstart;
    map.req = nullptr;
    map.n_vis = s_vcu[NI];
  } else {
    pdl_wait();  // use the validation kernel's prefix arrays
    if (!st->layout_ok) return;
    map.vcu = prep_vis_cu;
    map.gstart = nullptr;
    map.req = prep_img_req;
    map.n_vis = prep_vis_cu[NI];
    __syncwarp();
  }
  const uint64_t pol_first = policy_evict_first();
  const uint64_t pol_last = policy_evict_last();
  const int n_chunks = (D + kChunkElems - 1) / kChunkElems;
  const int64_t n_items = min(max(map.n_vis, int64_t(0)), T);  // visual ordinals (never more than T)
  // ---- work split. Each warp first takes a fixed contiguous run of whole tokens, about
  // 80 % of its even share; the rest of the tokens form a pool that the warps draw from
  // one token at a time (a counter the validation kernel resets), so that SMs with more
  // memory bandwidth take more of it and the CTAs finish together. Batches of fewer than
  // four tokens a warp are split evenly with no pool.
  // (visual ordinals are below 2^31: cu_seqlens are int32)
  const int32_t n_vis32 = static_cast<int32_t>(n_items);
  const int32_t n_warps = static_cast<int32_t>(gridDim.x) * kWarps;
  const int32_t gw = static_cast<int32_t>(blockIdx.x) * kWarps + warp;
  const bool pooled = n_items >= 4 * static_cast<int64_t>(n_warps);
  int32_t v_lo, v_hi, pool_lo;
  if (pooled) {
    const int32_t per = (n_vis32 - n_vis32 / 5) / n_warps;
    v_lo = gw * per;
    v_hi = v_lo + per;
    pool_lo = n_warps * per;
  } else {
    const int32_t per = n_vis32 / n_warps, extra = n_vis32 % n_warps;
    v_lo = gw * per + min(gw, extra);
    v_hi = v_lo + per + (gw < extra ? 1 : 0);
    pool_lo = n_vis32;
  }
  unsigned int* pool = &st->pool;
  bool waited = false;  // the validation kernel (which resets the pool and img_sums) is done
  auto wait_prep = [&]() {
    if (!waited) {
      pdl_wait();
      waited = true;
    }
  };
  // The next pool token is requested one token ahead (lane 0's atomic; its value is read
  // only when that token is due, so the request's latency hides behind the current one).
  bool pref = false;  // a request is outstanding (its value is in lane 0's pref_raw)
  unsigned int pref_raw = 0;
  auto request_pool = [&]() {
    wait_prep();
    if (lane == 0) pref_raw = atomicAdd(pool, 1u);
    pref = true;
  };
  // the token after `v` in this warp's sequence (n_items when there is none)
  auto next_token = [&](int32_t v) -> int32_t {
    if (v + 1 < v_hi) return v + 1;
    if (pool_lo >= n_vis32) return n_vis32;
    if (!pref) request_pool();
    const uint32_t k = __shfl_sync(0xffffffffu, pref_raw, 0);
    pref = false;
    return k < static_cast<uint32_t>(n_vis32 - pool_lo) ? pool_lo + static_cast<int32_t>(k) : n_vis32;
  };

  // issue side: token issue_v, chunk issue_chunk
  int32_t issue_v = v_lo < v_hi ? v_lo : next_token(v_hi - 1);
  int issue_chunk = 0;
  int issue_img = 0;
  int64_t issue_t = issue_v < n_vis32 ? map.position(issue_v, issue_img) : 0;
  // tokens issued (and the one prepared next) not yet consumed, oldest first: at most
  // kSlots + 1, when every token is one chunk
  int32_t q0 = issue_v, q1 = -1, q2 = -1, q3 = -1;
  if (issue_v < n_vis32 && issue_v + 1 >= v_hi && pool_lo < n_vis32) request_pool();

  auto issue_valid = [&]() { return issue_v < n_vis32; };
  auto advance_issue = [&]() {
    if (++issue_chunk < n_chunks) return;
    issue_chunk = 0;
    issue_v = next_token(issue_v);
    if (issue_v < n_vis32) {
      issue_t = map.position(issue_v, issue_img);
      if (q1 < 0) q1 = issue_v;
      else if (q2 < 0) q2 = issue_v;
      else q3 = issue_v;
      // starting the last fixed token, or a pool token: request the one after it
      if (issue_v + 1 >= v_hi && pool_lo < n_vis32 && !pref) request_pool();
    }
  };
  auto issue_one = [&](int slot) {
    const int e0 = issue_chunk * kChunkElems;
    const int ne = min(kChunkElems, D - e0);
    const uint32_t bytes = static_cast<uint32_t>(ne) * 2u;
    unsigned char* dst = wbuf + static_cast<size_t>(slot) * kSlotBytes;
    // a position outside [0, T) only comes from a malformed layout: read row 0 instead
    const int64_t t = (issue_t >= 0 && issue_t < T) ? issue_t : 0;
    if (lane == 0) {
      // order this warp's earlier shared-memory reads of the slot before the async-proxy writes
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_expect_tx(&wbar[slot], 2u * bytes);
      bulk_g2s(dst, h_cur + t * cur_stride + e0, bytes, &wbar[slot], pol_last);
      bulk_g2s(dst + kChunkBytes, h_prior + t * prior_stride + e0, bytes, &wbar[slot], pol_first);
    }
  };

  __syncwarp();
  uint32_t phase_bits = 0;  // bit s: parity to wait for on slot s
  int in_flight = 0;
  int slot_issue = 0;
  for (; in_flight < kSlots && issue_valid(); ++in_flight) {
    issue_one(slot_issue);
    slot_issue = (slot_issue + 1) % kSlots;
    advance_issue();
  }
  bool timed_out = false;
  // per lane: even and odd elements accumulate separately (one paired FMA each)
  float2 dot2 = make_float2(0.f, 0.f), na2 = dot2, nb2 = dot2;
  int slot_take = 0;
  int take_chunk = 0;
  int take_img = 0;
  int run_img = -1;     // image of the current run of rows (lane 0's view)
  int64_t run_sum = 0;  // its fixed-point sum so far
  auto add_to_image = [&](int img, int64_t v) {
    if (img_sums == nullptr) return;
    wait_prep();
    if (lane == 0) atomicAdd(reinterpret_cast<unsigned long long*>(img_sums + img), static_cast<unsigned long long>(v));
  };
  while (in_flight > 0) {
    const uint32_t parity = (phase_bits >> slot_take) & 1u;
    // warp-uniform bounded wait: a completed phase stays visible, so every lane gets there
    uint64_t t0 = 0;
    for (uint32_t polls = 1; !__all_sync(0xffffffffu, mbar_try_wait(&wbar[slot_take], parity)); ++polls) {
      if (__any_sync(0xffffffffu, wait_expired(polls, t0, kWaitLimitNs))) { timed_out = true; break; }
    }
    if (timed_out) break;
    phase_bits ^= 1u << slot_take;
    const int e0 = take_chunk * kChunkElems;
    const int ne = min(kChunkElems, D - e0);
    const uint4* a = reinterpret_cast<const uint4*>(wbuf + static_cast<size_t>(slot_take) * kSlotBytes);
    const uint4* b = reinterpret_cast<const uint4*>(wbuf + static_cast<size_t>(slot_take) * kSlotBytes + kChunkBytes);
    for (int c = lane; c < (ne >> 3); c += 32) {
      const uint4 va = a[c], vb = b[c];
      const uint32_t* pa = reinterpret_cast<const uint32_t*>(&va);
      const uint32_t* pb = reinterpret_cast<const uint32_t*>(&vb);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        // a bf16 pair widens to two fp32 values by placing each in the high half of a word
        const float2 fa = make_float2(__uint_as_float(pa[j] << 16), __uint_as_float(pa[j] & 0xffff0000u));
        const float2 fb = make_float2(__uint_as_float(pb[j] << 16), __uint_as_float(pb[j] & 0xffff0000u));
        dot2 = ffma2(fa, fb, dot2);
        na2 = ffma2(fa, fa, na2);
        nb2 = ffma2(fb, fb, nb2);
      }
    }
    __syncwarp();
    --in_flight;
    const bool row_done = take_chunk == n_chunks - 1;
    const int32_t take_v = q0;
    if (row_done) {  // the token leaves the queue before the refill may add one
      q0 = q1;
      q1 = q2;
      q2 = q3;
      q3 = -1;
    }
    // refill the slot just consumed
    if (issue_valid()) {
      issue_one(slot_take);
      advance_issue();
      ++in_flight;
    }
    slot_take = (slot_take + 1) % kSlots;
    if (row_done) {
      const float d = warp_sum(dot2.x + dot2.y), x = warp_sum(na2.x + na2.y), y = warp_sum(nb2.x + nb2.y);
      dot2 = na2 = nb2 = make_float2(0.f, 0.f);
      const int64_t t = map.position(take_v, take_img);
      const bool inside = t >= 0 && t < T;
      const float den = fmaxf(sqrtf(x), 1e-8f) * fmaxf(sqrtf(y), 1e-8f);
      const float I = 1.f - d / den;
      if (lane == 0 && inside) scores[t] = I;
      // run-length accumulation of the per-image sums (take_img is uniform over the warp)
      if (take_img != run_img) {
        if (run_img >= 0) add_to_image(run_img, run_sum);
        run_img = take_img;
        run_sum = 0;
      }
      if (inside) run_sum += fixed_point_score(I);
      take_chunk = 0;
    } else {
      ++take_chunk;
    }
  }
  if (!timed_out && run_img >= 0) add_to_image(run_img, run_sum);
  if (timed_out) {
    // drain: give the copies still in flight (slot_take and the in_flight - 1 slots after
    // it) a bounded chance to land before the CTA exits
    for (int k = 0; k < in_flight; ++k) {
      const int slot = (slot_take + k) % kSlots;
      const uint32_t parity = (phase_bits >> slot) & 1u;
      uint64_t t0 = 0;
      for (uint32_t polls = 1; !__all_sync(0xffffffffu, mbar_try_wait(&wbar[slot], parity)); ++polls)
        if (__any_sync(0xffffffffu, wait_expired(polls, t0, kWaitLimitNs))) break;
    }
    pdl_wait();  // the validation kernel resets the status word: record after it
    if (lane == 0) record_error(st, AVTP_ERR_TIMEOUT, static_cast<int32_t>(blockIdx.x));
  }
  pdl_wait();  // completion of this grid implies completion of the one before it
#ifdef AVTP_TIMELINE
  timeline_stamp_cta(st, kTlScoreEnd, &s_tl_done, kWarps);
#endif
}

}  // namespace

cudaError_t launch_score_hvar(const avtp_layout_t& L, const avtp_score_args_t& sa, float* scores,
                              int64_t* img_sums, void* ws, const WsPlan& p, cudaStream_t s, int reserve_sms) {
  if (L.n_images == 0 || L.n_tokens == 0) return cudaSuccess;
  // The dynamic shared memory a CTA may take: all an SM offers a CTA, less the static part.
  static PerDevice attrs;
  int smem_max = 0;
  cudaError_t ae = once_per_device(attrs, [](int dev, int* v) {
    int optin = 0;
    cudaFuncAttributes fa{};
    cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, k_score_hvar);
    if (e != cudaSuccess) return e;
    *v = optin - static_cast<int>(fa.sharedSizeBytes);
    if (*v < static_cast<int>(kSmemBytes)) return cudaErrorInvalidConfiguration;
    return cudaFuncSetAttribute(k_score_hvar, cudaFuncAttributeMaxDynamicSharedMemorySize, *v);
  }, &smem_max);
  if (ae != cudaSuccess) return ae;
  // With SMs left to the selection kernel, each scoring CTA takes all the shared memory a
  // CTA may have (the pipeline uses kSmemBytes of it): no CTA of the selection kernel can
  // then start next to it, so they all land on the free SMs. Sharing an SM with 16
  // streaming warps, a selection CTA fetched its code several times slower and its
  // warm-up run did not end before the scores did.
  const size_t smem = reserve_sms > 0 ? static_cast<size_t>(smem_max) : kSmemBytes;
  const int64_t want = (L.n_tokens + kWarps - 1) / kWarps;
  // one 192 KiB CTA per SM, except the SMs left to the next kernel
  int64_t cap = static_cast<int64_t>(device_sm_count()) - reserve_sms;
  if (cap < 1) cap = 1;
  const int grid = static_cast<int>(want < cap ? want : cap);
  cudaError_t e = launch_kernel(k_score_hvar, dim3(grid), dim3(kThreads), smem, s, /*pdl=*/true,
                                static_cast<const __nv_bfloat16*>(sa.h_cur), sa.h_cur_stride,
                                static_cast<const __nv_bfloat16*>(sa.h_prior), sa.h_prior_stride, sa.hidden,
                                L.cu_seqlens, L.n_requests, L.img_cu, L.img_start, L.img_len, L.n_images, L.n_tokens,
                                ws_at<int32_t>(ws, p.vis_cu), ws_at<int32_t>(ws, p.img_req), scores, img_sums,
                                ws_at<DevStatus>(ws, p.status));
  return e;
}

}  // namespace avtp
