// Step 4: compaction, out[j] = in[kept_idx[j]] for every row set (paper §3.1:
// E_pruned = p(E_v), the kept tokens as a dense, varlen-packed batch).
//
// Large rows (hidden states, K/V rows): one warp per row, 16-byte vector loads and
// stores; a lane issues all its loads of an 8-KiB piece of the row before its first
// store, so that a row costs one memory round trip (the scoring kernel reads h_cur with
// an evict-last policy, so some kept rows are still in L2). Small rows (position ids, one
// element per plane): one thread per row. All row sets go in one launch; the block index
// range is split between the sets on the host. A single-thread bulk-copy ring per SM
// (global -> shared -> global) was slower: the gather moves its bytes at about the HBM
// rate already, and one issuing thread per SM kept fewer of them in flight. So was a
// ring of bulk copies per warp with 192 KiB of slots per SM (the whole kept set in flight
// at once): 14.9 us against 11.7 us for this kernel on the Qwen3-VL-8B-shaped gather (28 MB
// of kept rows, h_cur read once beforehand, event-timed). Writing the 28 MB is the bound:
// a plain 28-MB fill takes about 12 us on this part.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRowsPerWarp = 1;
constexpr int kUnroll = 16;  // 16 x 16 bytes per lane: 8 KiB per warp in flight

struct RowSetDev {
  const char* in;
  char* out;
  int64_t row_bytes;
  int64_t in_stride;
  int64_t out_stride;
  int32_t unit;            // widest power-of-two access (1..16) dividing pointers, strides and row size
  int32_t warp_per_row;    // 1: vector path, one warp per row; 0: one thread per row
  int32_t rows_per_block;
  int32_t block_begin;
};

struct CompactParams {
  RowSetDev set[AVTP_MAX_ROW_SETS];
  int32_t n_sets;
};

template <int U>
struct UnitType;
template <> struct UnitType<16> { using T = uint4; };
template <> struct UnitType<8> { using T = uint2; };
template <> struct UnitType<4> { using T = uint32_t; };
template <> struct UnitType<2> { using T = uint16_t; };
template <> struct UnitType<1> { using T = uint8_t; };

template <int U>
__device__ __forceinline__ void copy_row_thread(const char* src, char* dst, int64_t bytes) {
  using T = typename UnitType<U>::T;
  const T* s = reinterpret_cast<const T*>(src);
  T* d = reinterpret_cast<T*>(dst);
  for (int64_t u = 0; u < bytes / U; ++u) d[u] = s[u];
}

__device__ __forceinline__ void compact_block(const CompactParams& P, int b, const int32_t* __restrict__ kept_idx,
                                              int64_t n_kept, int64_t n_tokens, DevStatus* st) {
  int si = 0;
  while (si + 1 < P.n_sets && b >= P.set[si + 1].block_begin) ++si;
  const RowSetDev S = P.set[si];
  const int64_t row0 = static_cast<int64_t>(b - S.block_begin) * S.rows_per_block;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (S.warp_per_row) {
    const int64_t n16 = S.row_bytes >> 4;
    for (int rr = 0; rr < kRowsPerWarp; ++rr) {
      const int64_t j = row0 + static_cast<int64_t>(rr) * kWarps + warp;
      if (j >= n_kept) break;
      const int64_t t = kept_idx[j];
      if (t < 0 || t >= n_tokens) {
        if (lane == 0) record_error(st, AVTP_ERR_DEVICE_INPUT, static_cast<int32_t>(j));
        continue;
      }
      const uint4* src = reinterpret_cast<const uint4*>(S.in + t * S.in_stride);
      uint4* dst = reinterpret_cast<uint4*>(S.out + j * S.out_stride);
      for (int64_t c0 = 0; c0 < n16; c0 += 32 * kUnroll) {
        uint4 v[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          const int64_t c = c0 + lane + 32 * u;
          if (c < n16) v[u] = __ldcs(src + c);
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          const int64_t c = c0 + lane + 32 * u;
          if (c < n16) __stcs(dst + c, v[u]);
        }
      }
    }
  } else {
    const int64_t j = row0 + threadIdx.x;
    if (static_cast<int>(threadIdx.x) >= S.rows_per_block || j >= n_kept) return;
    const int64_t t = kept_idx[j];
    if (t < 0 || t >= n_tokens) {
      record_error(st, AVTP_ERR_DEVICE_INPUT, static_cast<int32_t>(j));
      return;
    }
    const char* src = S.in + t * S.in_stride;
    char* dst = S.out + j * S.out_stride;
    switch (S.unit) {
      case 16: copy_row_thread<16>(src, dst, S.row_bytes); break;
      case 8: copy_row_thread<8>(src, dst, S.row_bytes); break;
      case 4: copy_row_thread<4>(src, dst, S.row_bytes); break;
      case 2: copy_row_thread<2>(src, dst, S.row_bytes); break;
      default: copy_row_thread<1>(src, dst, S.row_bytes); break;
    }
  }
}

// Grid-stride over the blocks of work (a block = kWarps rows of a vector set, or kThreads
// rows of a small set), with a grid the SMs hold at once: a second wave would start
// only when the first ends.
__global__ void __launch_bounds__(kThreads)
k_compact(CompactParams P, int n_blocks, const int32_t* __restrict__ kept_idx, int64_t n_kept, int64_t n_tokens,
          DevStatus* st) {
#ifdef AVTP_TIMELINE
  __shared__ unsigned s_tl_done;
  if (threadIdx.x == 0) {
    s_tl_done = 0;
    timeline_stamp(st, kTlCompactBegin);
  }
  __syncthreads();
#endif
  pdl_wait();  // kept_idx comes from the selection kernel
  pdl_trigger();
  if (threadIdx.x == 0) timeline_stamp(st, kTlCompactWaited);
  for (int b = blockIdx.x; b < n_blocks; b += gridDim.x) compact_block(P, b, kept_idx, n_kept, n_tokens, st);
#ifdef AVTP_TIMELINE
  timeline_stamp_cta(st, kTlCompactEnd, &s_tl_done, kWarps);
#endif
}

int compact_ctas_per_sm() {
  static PerDevice occ;
  int n = 0;
  const cudaError_t e = once_per_device(occ, [](int, int* v) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(v, k_compact, kThreads, 0);
  }, &n);
  return (e == cudaSuccess && n >= 1) ? n : 1;
}

int access_unit(const avtp_rows_t& s) {
  const uint64_t bits = reinterpret_cast<uint64_t>(s.in) | reinterpret_cast<uint64_t>(s.out) |
                        static_cast<uint64_t>(s.row_bytes) | static_cast<uint64_t>(s.in_stride) |
                        static_cast<uint64_t>(s.out_stride);
  for (int u = 16; u > 1; u >>= 1)
    if ((bits & static_cast<uint64_t>(u - 1)) == 0) return u;
  return 1;
}

}  // namespace

cudaError_t launch_compact(const int32_t* kept_idx, int64_t n_kept, int64_t n_tokens, const avtp_rows_t* sets,
                           int n_sets, void* ws, const WsPlan& p, cudaStream_t s) {
  if (n_kept == 0 || n_sets == 0) return cudaSuccess;
  CompactParams P{};
  P.n_sets = n_sets;
  int64_t blocks = 0;
  for (int i = 0; i < n_sets; ++i) {
    RowSetDev& d = P.set[i];
    d.in = static_cast<const char*>(sets[i].in);
    d.out = static_cast<char*>(sets[i].out);
    d.row_bytes = sets[i].row_bytes;
    d.in_stride = sets[i].in_stride;
    d.out_stride = sets[i].out_stride;
    d.unit = access_unit(sets[i]);
    d.warp_per_row = (d.unit == 16 && d.row_bytes >= 256) ? 1 : 0;
    d.rows_per_block = d.warp_per_row ? kWarps * kRowsPerWarp : kThreads;
    d.block_begin = static_cast<int32_t>(blocks);
    blocks += (n_kept + d.rows_per_block - 1) / d.rows_per_block;
  }
  if (blocks > 0x7fffffff) return cudaErrorInvalidConfiguration;
  const int64_t wave = static_cast<int64_t>(compact_ctas_per_sm()) * device_sm_count();
  const int64_t grid = blocks < wave ? blocks : wave;
  return launch_kernel(k_compact, dim3(static_cast<unsigned>(grid)), dim3(kThreads), 0, s, /*pdl=*/true, P,
                       static_cast<int>(blocks), kept_idx, n_kept, n_tokens, ws_at<DevStatus>(ws, p.status));
}

}  // namespace avtp
