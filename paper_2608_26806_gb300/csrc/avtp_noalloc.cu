// avtp_select_noalloc: the selection step for callers that cannot allocate
// device memory at the call site.
//
// Some callers cannot hand the library a workspace. An inference engine may
// reserve all free HBM for its KV-cache pool at start-up and pass plugins only
// their inputs and outputs. Code may run where allocation calls are not
// permitted, such as a host callback. For them this entry point keeps its
// scratch in a file-scope device array of fixed size, so no call to it
// allocates anything.
//
// The array has a fixed upper bound: AVTP_NOALLOC_MAX_IMAGES images and
// AVTP_NOALLOC_MAX_REQUESTS requests, about 145 KiB. Every GPU that loads this
// library holds it until the process exits. Calls share the array, and it
// keeps the contents of the last call; the validation kernel rewrites
// everything the selection kernel reads (status word, visual prefix, image ->
// request map) at the start of each call, so nothing stale is read. Two calls
// that overlap on the GPU (different streams, no ordering between them) race
// on the array and must not be issued.
#include "avtp_internal.cuh"

namespace avtp {
namespace {

constexpr size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

constexpr size_t kOffStatus = 0;
constexpr size_t kOffVisCu = align256(sizeof(DevStatus));
constexpr size_t kOffImgReq = kOffVisCu + align256(4 * (static_cast<size_t>(AVTP_NOALLOC_MAX_IMAGES) + 1));
constexpr size_t kOffReqBudget = kOffImgReq + align256(4 * static_cast<size_t>(AVTP_NOALLOC_MAX_IMAGES) + 4);
constexpr size_t kScratchBytes = kOffReqBudget + align256(4 * static_cast<size_t>(AVTP_NOALLOC_MAX_REQUESTS));

// The scratch itself. In host code this name is only a stand-in for the device
// array: its device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_select_scratch[kScratchBytes];

// Device address of the scratch on the current device. It is looked up on every call:
// the lookup allocates nothing, and an address cached across calls would go stale if
// the device's context were reset and the library's module reloaded elsewhere. The
// first lookup on a device may load the library's GPU module.
avtp_status_t scratch_for_current_device(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_select_scratch);
  if (e != cudaSuccess || p == nullptr) return AVTP_ERR_CUDA;
  *out = p;
  return AVTP_OK;
}

WsPlan scratch_plan() {
  WsPlan p{};
  p.status = kOffStatus;
  p.vis_cu = kOffVisCu;
  p.img_req = kOffImgReq;
  p.req_budget = kOffReqBudget;
  p.total = kScratchBytes;
  return p;
}

}  // namespace
}  // namespace avtp

using namespace avtp;

extern "C" avtp_status_t avtp_select_noalloc(const avtp_layout_t* layout, const float* scores,
                                             const int32_t* budgets, const int32_t* out_cu_seqlens,
                                             int32_t* kept_idx, int64_t n_kept, int32_t* device_status,
                                             avtp_stream_t stream) {
  if (layout == nullptr) return AVTP_ERR_INVALID_ARG;
  const avtp_layout_t& L = *layout;
  if (L.n_requests < 1 || L.n_images < 0 || L.n_tokens < 0) return AVTP_ERR_INVALID_ARG;
  if (L.n_tokens > 0x7fffffffLL) return AVTP_ERR_RANGE;
  if (L.n_images > AVTP_NOALLOC_MAX_IMAGES || L.n_requests > AVTP_NOALLOC_MAX_REQUESTS) return AVTP_ERR_RANGE;
  if (L.cu_seqlens == nullptr || L.img_cu == nullptr) return AVTP_ERR_INVALID_ARG;
  if (L.n_images > 0 && (L.img_start == nullptr || L.img_len == nullptr || scores == nullptr || budgets == nullptr))
    return AVTP_ERR_INVALID_ARG;
  if (out_cu_seqlens == nullptr || n_kept < 0 || (n_kept > 0 && kept_idx == nullptr)) return AVTP_ERR_INVALID_ARG;
  void* ws = nullptr;
  avtp_status_t st = scratch_for_current_device(&ws);
  if (st != AVTP_OK) return st;
  const WsPlan p = scratch_plan();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PrepArgs pa{};
  pa.L = L;
  if (launch_prep(pa, ws, p, s) != cudaSuccess) return AVTP_ERR_CUDA;
  if (launch_select(L, scores, budgets, out_cu_seqlens, kept_idx, n_kept, ws, p, s) != cudaSuccess)
    return AVTP_ERR_CUDA;
  if (device_status != nullptr &&
      cudaMemcpyAsync(device_status, static_cast<char*>(ws) + p.status, sizeof(int32_t), cudaMemcpyDeviceToDevice,
                      s) != cudaSuccess)
    return AVTP_ERR_CUDA;
  return AVTP_OK;
}
