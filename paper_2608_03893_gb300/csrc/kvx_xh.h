// Pieces of the cross-head path (kvx_xh.cu) shared with the MLP mapper (kvx_mlp.cu).
#pragma once

#include "kvx_internal.h"

namespace kvx {

// Source keys with the source RoPE stripped and rounded to bf16, written contiguously as
// [L_s][B][H][T][128] into `ws`; `ss` the source strides (layer, batch, head, token);
// `hf`: the Hugging Face forward's rounding (kvx_rope_numerics); `il`: interleaved RoPE
// pairs (2i, 2i+1) instead of half-split pairs (i, i + 64).
void launch_key_strip(const void* src_k, const int64_t* ss, void* ws, const int32_t* pos, int Ls, int H, int B, int T,
                      const RopeTables& rope, int sms, cudaStream_t stream, int hf, int il);

// fp32 W [L_t][2][H][F][128] -> W^T bf16 [L_t][2][H][128][2F] = [W_hi | W_lo] in ctx->d_Wt,
// for the tensor-core map kernels (cross-head and per-head) with fp32 weights.
kvx_status repack_wt_hilo(kvx_ctx* c, const void* W_host, size_t F);

}  // namespace kvx
