// Pruning-layer selection (paper §3.3.2): for N sample requests run through an LVLM, the
// attention each layer l assigns to the visual tokens, A_l^(i) = sum_j Attention(l, v_j),
// the rank of every layer within each sample, the average rank R_l over the samples, and
// the k layers with the best average rank as the pruning layers.
//
// k_layer_attention: A[r][layer] = sum of the request's fixed-point image sums of the
// text-attention criterion at that layer (units of 2^-32, exact integers), a warp per
// request. Called once per layer, it fills one column of A.
// k_layer_select: one CTA. Rank(A_l^(i)) = 1 + #{l' : A_l' > A_l} + #{l' < l : A_l' = A_l}
// (1 for the most attention, equal values to the lower layer), summed over the samples
// with integer atomics in shared memory (order-independent); then each layer's place
// among the rank sums (ties to the lower layer) puts the best k in top_layers.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kSelThreads = 1024;

__global__ void __launch_bounds__(256)
k_layer_attention(const int32_t* __restrict__ img_cu, int R, const int64_t* __restrict__ img_sums,
                  int64_t* __restrict__ A, int n_layers, int layer, const DevStatus* st) {
  pdl_wait();
  pdl_trigger();
  if (!st->layout_ok) return;
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < R; r += warps) {
    int64_t s = 0;
    for (int i = img_cu[r] + lane; i < img_cu[r + 1]; i += 32) s += img_sums[i];
    s = warp_sum(s);
    if (lane == 0) A[static_cast<int64_t>(r) * n_layers + layer] = s;
  }
}

__global__ void __launch_bounds__(kSelThreads)
k_layer_select(const int64_t* __restrict__ A, int N, int L, int k, int64_t* __restrict__ rank_sum,
               int32_t* __restrict__ top_layers) {
  __shared__ unsigned long long s_rank[AVTP_MAX_LAYERS];
  pdl_wait();
  pdl_trigger();
  for (int l = threadIdx.x; l < L; l += blockDim.x) s_rank[l] = 0ull;
  __syncthreads();
  const int64_t pairs = static_cast<int64_t>(N) * L;
  for (int64_t u = threadIdx.x; u < pairs; u += blockDim.x) {
    const int i = static_cast<int>(u / L), l = static_cast<int>(u % L);
    const int64_t* row = A + static_cast<int64_t>(i) * L;
    const int64_t a = row[l];
    unsigned long long rank = 1;
    for (int m = 0; m < L; ++m) {
      const int64_t b = row[m];
      rank += (b > a || (b == a && m < l)) ? 1ull : 0ull;
    }
    atomicAdd(&s_rank[l], rank);
  }
  __syncthreads();
  for (int l = threadIdx.x; l < L; l += blockDim.x) {
    const unsigned long long rl = s_rank[l];
    rank_sum[l] = static_cast<int64_t>(rl);
    int place = 0;
    for (int m = 0; m < L; ++m) {
      const unsigned long long rm = s_rank[m];
      place += (rm < rl || (rm == rl && m < l)) ? 1 : 0;
    }
    if (place < k) top_layers[place] = l;
  }
}

}  // namespace

cudaError_t launch_layer_attention(const avtp_layout_t& L, const int64_t* img_sums, int64_t* A, int n_layers,
                                   int layer, void* ws, const WsPlan& p, cudaStream_t s) {
  const int64_t want = (static_cast<int64_t>(L.n_requests) * 32 + 255) / 256;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 4;
  const int grid = static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
  return launch_kernel(k_layer_attention, dim3(grid), dim3(256), 0, s, /*pdl=*/true, L.img_cu, L.n_requests,
                       img_sums, A, n_layers, layer, static_cast<const DevStatus*>(ws_at<DevStatus>(ws, p.status)));
}

cudaError_t launch_layer_select(const int64_t* A, int n_samples, int n_layers, int k, int64_t* rank_sum,
                                int32_t* top_layers, cudaStream_t s) {
  return launch_kernel(k_layer_select, dim3(1), dim3(kSelThreads), 0, s, /*pdl=*/false, A, n_samples, n_layers, k,
                       rank_sum, top_layers);
}

}  // namespace avtp
