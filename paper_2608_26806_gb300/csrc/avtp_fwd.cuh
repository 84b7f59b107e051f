// Host-side declarations of the layer's causal attention forward (k_attn_fwd.cu).
#pragma once

#include "avtp_internal.cuh"

namespace avtp {

// Workspace of avtp_attn_forward beyond the criterion-B part (which is the plan of
// plan_workspace with the forward's LSE supplied).
struct FwdWs {
  size_t vt;        // bf16 [Hkv][d][Tp]: the values transposed, tokens contiguous
  size_t qtile_cu;  // int32 [R + 1]: query tiles of 128 tokens per request, prefix
  int64_t Tp;       // T rounded up to a multiple of 8 (16-byte rows of vt)
  size_t total;
};
FwdWs plan_forward_workspace(const avtp_layout_t& L, const avtp_score_args_t& sa, size_t base_bytes);

// The forward proper: transposed values, query-tile prefix, then the tcgen05 kernel that
// writes O and the natural-log LSE.
cudaError_t launch_attn_forward(const avtp_layout_t& L, const avtp_score_args_t& sa, const avtp_forward_args_t& fa,
                                void* ws, const WsPlan& p, const FwdWs& f, cudaStream_t s);

}  // namespace avtp
