// Internal declarations shared by the host library and the kernels of libkvx.
#pragma once

#include <cstdint>
#include <string>
#include <vector>

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "../../include/kvx.h"

namespace kvx {

// A named NVTX range over one entry point's host work (its launches and copies show
// under it in a timeline profiler); a no-op unless a profiler is attached.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

constexpr int kMaxHeadDim = 256;
constexpr int kMaxPairs = kMaxHeadDim / 2;

// RoPE inverse frequencies omega_i = theta^(-2i/d) as an unevaluated sum hi + lo of two
// floats (hi = fl32(omega), lo = fl32(omega - hi)), plus the two-float split of 2*pi
// used to reduce t * omega into [-pi, pi] with fused multiply-adds (Cody-Waite).
struct RopeTables {
  float ws_hi[kMaxPairs], ws_lo[kMaxPairs];  // source theta
  float wt_hi[kMaxPairs], wt_lo[kMaxPairs];  // target theta
  float two_pi_hi, two_pi_lo, inv_two_pi;
};

// Everything a kernel needs about one kvx_map call.
struct MapArgs {
  const void* src_k;
  const void* src_v;
  int64_t ss[4];            // source strides (layer, batch, head, token), elements
  void* tgt_k;
  void* tgt_v;
  int64_t ts[4];            // target strides (layer, batch|block, head, token|slot)
  int32_t paged, block_size, max_blocks, n_blocks;
  const int32_t* block_table;
  const int32_t* pos;       // [B][T]
  int32_t B, T;
};

// Tensor-core plan: a schedule of source-tile loads into a ring of shared-memory slots,
// the same for every work unit (it depends only on the selection table).  Uses are the
// (target layer l, selection j) pairs in l-major order.
struct TcPlan {
  int32_t n_slots = 0;                  // source-tile slots (tensor memory)
  int32_t n_land = 0;                   // source landing buffers in shared memory
  int32_t n_wst = 0;                    // W stages in shared memory
  int32_t n_loads = 0;                  // source-tile loads per work unit
  std::vector<int32_t> load_layer;      // [n_loads] source layer of load e
  std::vector<int32_t> load_slot;       // [n_loads] slot it lands in
  std::vector<int32_t> load_first_use;  // [n_loads] target layer of its first use
  std::vector<int32_t> use_slot;        // [L_t*k] slot holding the tile of use (l, j)
  std::vector<int32_t> use_flags;       // [L_t*k] bit 0: first use of the tile by its issuer,
                                        //         bit 2: release the slot after this use
};

}  // namespace kvx

struct kvx_ctx {
  int device = 0;
  int Ls = 0, Lt = 0, H = 0, d = 0, k = 0, F = 0;
  int rope_style = 0, cache_dtype = 0, weight_dtype = 0, head_mix = 0;
  double theta_s = 0, theta_t = 0;
  int rope_numerics = 0;                          // kvx_rope_numerics
  bool scale_s_on = false, scale_t_on = false;   // Llama-3 frequency scaling per side
  kvx_rope_scaling scale_s{}, scale_t{};
  int kernel = KVX_KERNEL_AUTO;
  bool tc_eligible = false;
  bool xh_eligible = false;         // cross-head tensor-core kernel
  std::vector<int32_t> sel;          // host copy [L_t][k]
  kvx::RopeTables rope{};
  // device memory owned by the context
  int32_t* d_sel = nullptr;          // [L_t][k]
  void* d_W = nullptr;               // [L_t][2][H][F][d] as given (SIMT kernel)
  float* d_b = nullptr;              // [L_t][2][H][d] fp32 (zeros when b == NULL)
  void* d_Wt = nullptr;              // tensor-core layout (bf16), see kvx_tc.cu
  int32_t* d_plan = nullptr;         // tensor-core schedule tables
  int32_t* d_status = nullptr;       // device status word
  void* d_ws = nullptr;              // cross-head kernel: source keys with the RoPE stripped
  size_t ws_bytes = 0;
  kvx::TcPlan plan;
  int sm_count = 0;
  // test switches (kvx_set_test_wait): the per-head tensor-core kernel's wait bound, and a
  // bias row its first CTA never loads, which makes one of its waits run out
  int F_xh = 0;                      // feature width of the cross-head kernel's W^T: F for a
                                     // cross-head mapper, k * H * d for a per-head one (block-
                                     // diagonal W, zero outside head h's rows)
  uint64_t wait_limit_ns = 0;        // 0: the default bound
  int64_t skip_bias_row = -1;
};

namespace kvx {
void set_error(const std::string& msg);

// NULL if the scaling (or NULL) is valid, else why not.
const char* check_rope_scaling(const kvx_rope_scaling* s);
// Copies the two optional scalings into the context (after check_rope_scaling).
void set_rope_scaling(kvx_ctx* c, const kvx_rope_scaling* src, const kvx_rope_scaling* tgt);

// Fills ctx->rope from ctx->d, ctx->theta_s, ctx->theta_t and the optional scalings.
void fill_rope(kvx_ctx* c);

// SIMT fp32 kernel (any head_dim <= 256, fp32 or bf16 caches/weights, both layouts).
kvx_status launch_simt(const kvx_ctx* ctx, const MapArgs& a, cudaStream_t stream);

// Tensor-core kernel (bf16, head_dim 128, per-head, half-split pairs).
bool tc_supported(const kvx_ctx* ctx, std::string* why);
kvx_status tc_prepare(kvx_ctx* ctx, const void* W_host);   // repack W, build the plan
kvx_status launch_tc(const kvx_ctx* ctx, const MapArgs& a, cudaStream_t stream);
// W [L_t][2][H][F][d] -> W^T [L_t][2][H][d][F] bf16 in ctx->d_Wt (both tensor-core kernels).
kvx_status repack_wt(kvx_ctx* ctx, const void* W_host, size_t F);
// cuTensorMapEncodeTiled from the driver (as void*: PFN_cuTensorMapEncodeTiled_v12000), or NULL.
void* tensor_map_encoder();

// Tensor-core kernel for the cross-head feature layout (bf16, head_dim 128, half-split
// pairs, even head count, contiguous targets): a source-key RoPE strip into a workspace,
// then one pair-MMA GEMM per (target layer, K|V).
bool xh_supported(const kvx_ctx* ctx, std::string* why);
kvx_status launch_xh(kvx_ctx* ctx, const MapArgs& a, cudaStream_t stream);

}  // namespace kvx
