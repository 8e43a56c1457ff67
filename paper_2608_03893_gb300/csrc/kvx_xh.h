// Pieces of the cross-head path (kvx_xh.cu) shared with the MLP mapper (kvx_mlp.cu).
#pragma once

#include "kvx_internal.h"

namespace kvx {

// Source keys with the source RoPE stripped and rounded to bf16, written contiguously as
// [L_s][B][H][T][128] into `ws`; `ss` the source strides (layer, batch, head, token).
void launch_key_strip(const void* src_k, const int64_t* ss, void* ws, const int32_t* pos, int Ls, int H, int B, int T,
                      const RopeTables& rope, int sms, cudaStream_t stream);

}  // namespace kvx
