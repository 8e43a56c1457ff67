// MLP mapper apply (Sec. 4.3, Appendix "Run information"): per target layer l, K|V and
// head h,
//   y = W3 relu(W2 relu(W1 x + b1) + b2) + b3     (nn.Linear convention, weights [out][in]),
// x the cross-head source feature (the k selected source layers' heads, head-minor; keys
// RoPE-stripped and rounded to bf16, as in the ridge path), keys re-rotated with the target
// RoPE after the bias, bf16 out.  Each hidden activation is stored in bf16 after its ReLU.
//
// Three GEMM passes per group of target layers, each one launch of tc_mlp_kernel (clusters
// of two CTAs, pair MMAs cta_group::2 with M = 256 tokens, operands in shared memory by TMA
// in three 64 KB stages of 128 features, fp32 accumulators in TMEM):
//   pass 1: H1[l,kv] = relu(X_l W1[l,kv,:]^T + b1)  -- one GEMM per (l, K|V) over all heads'
//           hidden units (N = H hidden), K = k H d; A tiles straight from the stripped-key
//           workspace / the value cache (5-D TMA, as the cross-head ridge kernel);
//   pass 2: H2[l,kv,h] = relu(H1[l,kv,h] W2[l,kv,h]^T + b2), K = N = hidden;
//   pass 3: y[l,kv,h] = H2[l,kv,h] W3[l,kv,h]^T + b3 (N = 128), target RoPE, bf16 store.
// H1 and H2 live in a workspace [group layer][K|V][token][H hidden] bf16.  Work unit =
// (output tile of 256 columns, head, pair of 128-token tiles, sequence, K|V, layer), the
// output tile fastest so the clusters in flight share the A tiles of one token-tile pair.
// Roles (384 threads): warp 0 TMA producer, warp 1 TMEM allocator and (rank 0) MMA issuer
// (eight MMAs per stage), warps 4-11 epilogue (two warpgroups: columns 0-127 and 128-255 of
// a tile; in pass 3 RoPE pairs 0-31 and 32-63).  Every wait is bounded (KVX_ERR_TIMEOUT).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <cstring>
#include <string>

#include "kvx_internal.h"
#include "kvx_ptx.cuh"
#include "kvx_rope.cuh"
#include "kvx_xh.h"

namespace kvx {
namespace {

using namespace ptx;

constexpr int kMThreads = 384;
constexpr int kMFirstEpi = 4;
constexpr int kMEpiWarps = 8;
constexpr int kMD = 128;                          // head_dim
constexpr int kMTile = 128;                       // tokens per CTA
constexpr int kMStages = 3;
constexpr uint32_t kMABytes = kMTile * 128 * 2;   // 128 tokens x 128 features (two 64-wide halves), 32 KB
constexpr uint32_t kMBBytes = 128 * 128 * 2;      // 128 output rows x 128 features (two halves), 32 KB
constexpr uint32_t kMStageBytes = kMABytes + kMBBytes;
constexpr uint32_t kMAccCols = 256;
constexpr uint32_t kMTmemCols = 512;
constexpr size_t kMSmemLimit = 232448;

constexpr size_t mlp_smem_bytes() {
  return static_cast<size_t>(kMStages) * kMStageBytes + (2 * kMStages + 4 + 1) * 8 + 16;
}
static_assert(mlp_smem_bytes() <= kMSmemLimit, "MLP kernel shared memory exceeds the per-CTA limit");

struct MlpParams {
  CUtensorMap tm_ak;       // pass 1 A: stripped keys [L_s][B][H][T][128], box 64 x 128
  CUtensorMap tm_av;       // pass 1 A: source values (caller's strides), box 64 x 128
  CUtensorMap tm_h;        // passes 2, 3 A: hidden input [rows = G 2 N][H hidden], box 64 x 128
  CUtensorMap tm_w;        // B: the pass's weights [rows][K], box 64 x 128 (pass 3: 64 x 64)
  const float* bias;       // the pass's bias, [L_t][2][n_out_total]
  __nv_bfloat16* hout;     // passes 1, 2: hidden output [G 2 N][H hidden]
  MapArgs a;               // positions, targets (pass 3), B, T
  const int32_t* sel;      // [L_t][k]
  int32_t* status;
  int32_t pass, l0, H, k, hidden, pairs, n_units, n_tiles, heads, ksteps, G, hf;
  RopeTables rope;
};

struct MUnit {
  int nt, h, t0, b, kv, lg;
};

// Unit order: output tile fastest, then head, token-tile pair, sequence, K|V, group layer.
__device__ __forceinline__ MUnit mlp_decode(int u, const MlpParams& P, uint32_t rank) {
  MUnit r;
  r.nt = u % P.n_tiles;
  int rest = u / P.n_tiles;
  r.h = rest % P.heads;
  rest /= P.heads;
  r.t0 = (2 * (rest % P.pairs) + static_cast<int>(rank)) * kMTile;
  rest /= P.pairs;
  r.b = rest % P.a.B;
  rest /= P.a.B;
  r.kv = rest % 2;
  r.lg = rest / 2;
  return r;
}

__device__ __forceinline__ void mreport(int32_t* status, int code) { atomicCAS(status, 0, code); }

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kMThreads, 1)
    tc_mlp_kernel(const __grid_constant__ MlpParams P) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) mreport(P.status, KVX_ERR_UNSUPPORTED);
    return;
  }
  uint8_t* stages = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(kMStages) * kMStageBytes);
  uint64_t* empty = full + kMStages;
  uint64_t* accf = empty + kMStages;       // [2] accumulator ready (both CTAs)
  uint64_t* acce = accf + 2;               // [2] accumulator drained (8 warps x 2 CTAs, rank 0)
  uint64_t* drain = acce + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  volatile uint32_t* abort_flag = tmem_holder + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int unit0 = blockIdx.x >> 1, unit_step = gridDim.x >> 1;
  const bool narrow = P.pass == 3;         // N = 128: each CTA holds 64 rows of B
  const uint32_t b_bytes = narrow ? kMBBytes / 2 : kMBBytes;
  const uint32_t b_half = b_bytes / 2;     // one 64-feature half of B

  if (threadIdx.x == 0) {
    for (int i = 0; i < kMStages; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accf[i]), 1);
      mbar_init(smem_u32(&acce[i]), 2 * kMEpiWarps);
    }
    mbar_init(smem_u32(&drain[0]), 1);
    *abort_flag = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(kMTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int n_units = P.n_units, ksteps = P.ksteps, H = P.H;
  const int64_t N = static_cast<int64_t>(P.a.B) * P.a.T;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer ----
    if (lane == 0) {
      const uint64_t pol_a = policy_evict_last();
      const uint64_t pol_w = policy_evict_last();
      uint32_t sn = 0;
      bool ok = true;
      for (int u = unit0; ok && u < n_units; u += unit_step) {
        const MUnit un = mlp_decode(u, P, rank);
        const int l = P.l0 + un.lg;
        for (int s = 0; s < ksteps; ++s, ++sn) {
          const int st = static_cast<int>(sn % kMStages);
          const uint32_t round = sn / kMStages;
          if (round > 0 &&
              !wait_bar(smem_u32(&empty[st]), (round - 1) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT)) {
            ok = false;
            break;
          }
          if (rank == 0) mbar_expect_tx(smem_u32(&full[st]), 2 * (kMABytes + b_bytes));
          const uint32_t bar = mapa_shared(smem_u32(&full[st]), 0);
          const uint32_t a_dst = smem_u32(stages + static_cast<size_t>(st) * kMStageBytes);
          const uint32_t b_dst = a_dst + kMABytes;
          int wrow;
          if (P.pass == 1) {
            // feature block s: source layer sel[l][s / H], head s % H
            const int j = s / H, hs = s % H;
            const int L = __ldg(&P.sel[l * P.k + j]);
            const CUtensorMap* tm = un.kv ? &P.tm_av : &P.tm_ak;
            tma_load_5d_pair(a_dst, tm, bar, 0, un.t0, hs, un.b, L, pol_a);
            tma_load_5d_pair(a_dst + kMABytes / 2, tm, bar, 64, un.t0, hs, un.b, L, pol_a);
            wrow = (l * 2 + un.kv) * H * P.hidden + un.nt * 256;
          } else {
            const int row = static_cast<int>((static_cast<int64_t>(un.lg) * 2 + un.kv) * N +
                                             static_cast<int64_t>(un.b) * P.a.T + un.t0);
            tma_load_2d_pair(a_dst, &P.tm_h, bar, un.h * P.hidden + 128 * s, row, pol_a);
            tma_load_2d_pair(a_dst + kMABytes / 2, &P.tm_h, bar, un.h * P.hidden + 128 * s + 64, row, pol_a);
            wrow = P.pass == 2 ? ((l * 2 + un.kv) * H + un.h) * P.hidden + un.nt * 256
                               : ((l * 2 + un.kv) * H + un.h) * kMD;
          }
          const int brow = wrow + static_cast<int>(rank) * (narrow ? 64 : 128);
          tma_load_2d_pair(b_dst, &P.tm_w, bar, 128 * s, brow, pol_w);
          tma_load_2d_pair(b_dst + b_half, &P.tm_w, bar, 128 * s + 64, brow, pol_w);
        }
      }
      if (!ok && rank == 0) {   // the most recent loads may still be landing
        const uint32_t first = sn > static_cast<uint32_t>(kMStages) ? sn - kMStages : 0;
        for (uint32_t i = first; i < sn; ++i) drain_wait(smem_u32(&full[i % kMStages]), (i / kMStages) & 1u);
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer ----
    if (lane == 0 && rank == 0) {
      const uint32_t idesc = narrow ? make_idesc(2 * kMTile, 128) : make_idesc(2 * kMTile, 256);
      uint32_t si = 0, acc_n = 0;
      bool ok = true, issued = false;
      for (int u = unit0; ok && u < n_units; u += unit_step, ++acc_n) {
        const uint32_t buf = acc_n & 1u;
        if (acc_n >= 2 && !wait_bar(smem_u32(&acce[buf]), ((acc_n >> 1) - 1) & 1u, abort_flag, P.status,
                                    KVX_ERR_TIMEOUT)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + buf * kMAccCols;
        for (int s = 0; s < ksteps; ++s, ++si) {
          const uint32_t st = si % kMStages;
          if (!wait_bar(smem_u32(&full[st]), (si / kMStages) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(stages + static_cast<size_t>(st) * kMStageBytes);
          const uint32_t b0 = a0 + kMABytes;
#pragma unroll
          for (int half = 0; half < 2; ++half)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_ss_pair(d_tmem, sw128_desc(a0 + half * (kMABytes / 2) + kk * 32),
                             sw128_desc(b0 + half * b_half + kk * 32), idesc, (s | half | kk) != 0);
          issued = true;
          tc_commit_pair(smem_u32(&empty[st]), 3);
        }
        if (ok) tc_commit_pair(smem_u32(&accf[buf]), 3);
      }
      if (issued || !ok) {
        tc_commit_pair(smem_u32(&drain[0]), 1);
        drain_wait(smem_u32(&drain[0]), 0);
      }
    }
  } else if (warp >= kMFirstEpi) {
    // -------------------------------------------------------------- epilogue ------
    const int g = (warp - kMFirstEpi) >> 2;          // warpgroup: columns 128g.. (pass 3: pairs 32g..)
    const int q = warp & 3;                          // TMEM lane quarter
    const int r = q * 32 + lane;                     // token row within the tile
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    const uint64_t st_pol = policy_evict_first();
    uint32_t acc_n = 0;
    float cs[32], sn[32];
    for (int u = unit0; u < n_units; u += unit_step, ++acc_n) {
      const MUnit un = mlp_decode(u, P, rank);
      const int l = P.l0 + un.lg;
      const int t = un.t0 + r;
      bool valid = t < P.a.T;
      const uint32_t buf = acc_n & 1u;
      const bool w_ok = wait_bar(smem_u32(&accf[buf]), (acc_n >> 1) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT);
      if (!__all_sync(0xffffffffu, w_ok)) break;
      tc_fence_after();
      const uint32_t col0 = tmem_base + lane_addr + buf * kMAccCols;
      if (P.pass != 3) {
        // 128 columns of this warpgroup: + bias, ReLU, bf16, stored to the hidden workspace
        const int n_out = P.pass == 1 ? H * P.hidden : P.hidden;
        const int c0 = un.nt * 256 + 128 * g;        // column within the (l, kv[, h]) block
        const float* bias = P.bias + static_cast<size_t>(l * 2 + un.kv) * H * P.hidden +
                            (P.pass == 2 ? un.h * P.hidden : 0) + c0;
        __nv_bfloat16* out = P.hout + ((static_cast<int64_t>(un.lg) * 2 + un.kv) * N +
                                       static_cast<int64_t>(un.b) * P.a.T + t) * (static_cast<int64_t>(H) * P.hidden) +
                             (P.pass == 2 ? un.h * P.hidden : 0) + c0;
        (void)n_out;
#pragma unroll 1
        for (int c = 0; c < 128; c += 32) {
          uint32_t lo[16], hi[16];
          tmem_ld_2x16(col0 + 128 * g + c, col0 + 128 * g + c + 16, lo, hi);
          if (c == 96) {   // the accumulator is free for the unit after next
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&acce[buf]), 0));
          }
          uint32_t w[16];
#pragma unroll
          for (int e = 0; e < 16; e += 4) {
            const float4 bl = __ldg(reinterpret_cast<const float4*>(bias + c + e));
            const float4 bh = __ldg(reinterpret_cast<const float4*>(bias + c + 16 + e));
            w[e / 2] = pack_bf16x2(fmaxf(__fadd_rn(__uint_as_float(lo[e]), bl.x), 0.f),
                                   fmaxf(__fadd_rn(__uint_as_float(lo[e + 1]), bl.y), 0.f));
            w[e / 2 + 1] = pack_bf16x2(fmaxf(__fadd_rn(__uint_as_float(lo[e + 2]), bl.z), 0.f),
                                       fmaxf(__fadd_rn(__uint_as_float(lo[e + 3]), bl.w), 0.f));
            w[8 + e / 2] = pack_bf16x2(fmaxf(__fadd_rn(__uint_as_float(hi[e]), bh.x), 0.f),
                                       fmaxf(__fadd_rn(__uint_as_float(hi[e + 1]), bh.y), 0.f));
            w[8 + e / 2 + 1] = pack_bf16x2(fmaxf(__fadd_rn(__uint_as_float(hi[e + 2]), bh.z), 0.f),
                                           fmaxf(__fadd_rn(__uint_as_float(hi[e + 3]), bh.w), 0.f));
          }
          if (valid) {
#pragma unroll
            for (int v = 0; v < 4; ++v)
              st_global_hint(out + c + 8 * v, make_uint4(w[4 * v], w[4 * v + 1], w[4 * v + 2], w[4 * v + 3]),
                             st_pol);
          }
        }
      } else {
        // pass 3: 32 RoPE pairs (channels 32g.. and 64+32g..) + bias, target RoPE, bf16
        int p = 0;
        if (valid) {
          p = __ldg(&P.a.pos[static_cast<int64_t>(un.b) * P.a.T + t]);
          if (p < 0 || p >= (1 << 24)) {
            mreport(P.status, KVX_ERR_DEVICE_BOUNDS);
            valid = false;
            p = 0;
          }
        }
        if (un.kv == 0 && P.hf) {   // HF numerics: cos / sin of the fp32 angle, rounded to bf16
#pragma unroll
          for (int m = 0; m < 32; ++m) {
            sincosf(__fmul_rn(static_cast<float>(p), P.rope.wt_hi[32 * g + m]), &sn[m], &cs[m]);
            sn[m] = __bfloat162float(__float2bfloat16_rn(sn[m]));
            cs[m] = __bfloat162float(__float2bfloat16_rn(cs[m]));
          }
        } else if (un.kv == 0) {
#pragma unroll
          for (int m = 0; m < 32; ++m)
            rope_sincos(p, P.rope.wt_hi[32 * g + m], P.rope.wt_lo[32 * g + m], P.rope.two_pi_hi, P.rope.two_pi_lo,
                        P.rope.inv_two_pi, &sn[m], &cs[m]);
        }
        const float* bias = P.bias + (static_cast<size_t>(l * 2 + un.kv) * H + un.h) * kMD;
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(un.kv ? P.a.tgt_v : P.a.tgt_k) +
                             static_cast<int64_t>(l) * P.a.ts[0] + un.b * P.a.ts[1] +
                             static_cast<int64_t>(un.h) * P.a.ts[2] + static_cast<int64_t>(t) * P.a.ts[3];
#pragma unroll
        for (int rnd = 0; rnd < 2; ++rnd) {
          uint32_t lo[16], hi[16];
          const uint32_t col = col0 + 32 * g + 16 * rnd;
          tmem_ld_2x16(col, col + 64, lo, hi);
          if (rnd == 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&acce[buf]), 0));
          }
          const int c_lo = 32 * g + 16 * rnd;
          float ylo[16], yhi[16];
#pragma unroll
          for (int j = 0; j < 16; j += 4) {
            const float4 b0 = __ldg(reinterpret_cast<const float4*>(bias + c_lo + j));
            const float4 b1 = __ldg(reinterpret_cast<const float4*>(bias + 64 + c_lo + j));
            ylo[j] = __fadd_rn(__uint_as_float(lo[j]), b0.x);
            ylo[j + 1] = __fadd_rn(__uint_as_float(lo[j + 1]), b0.y);
            ylo[j + 2] = __fadd_rn(__uint_as_float(lo[j + 2]), b0.z);
            ylo[j + 3] = __fadd_rn(__uint_as_float(lo[j + 3]), b0.w);
            yhi[j] = __fadd_rn(__uint_as_float(hi[j]), b1.x);
            yhi[j + 1] = __fadd_rn(__uint_as_float(hi[j + 1]), b1.y);
            yhi[j + 2] = __fadd_rn(__uint_as_float(hi[j + 2]), b1.z);
            yhi[j + 3] = __fadd_rn(__uint_as_float(hi[j + 3]), b1.w);
          }
          if (un.kv == 0 && P.hf) {   // the key as a bf16 tensor, each product and sum rounded
            auto r = [](float x) { return __bfloat162float(__float2bfloat16_rn(x)); };
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float c = cs[16 * rnd + j], s = sn[16 * rnd + j];
              const float y0 = r(ylo[j]), y1 = r(yhi[j]);
              ylo[j] = r(__fsub_rn(r(__fmul_rn(y0, c)), r(__fmul_rn(y1, s))));
              yhi[j] = r(__fadd_rn(r(__fmul_rn(y1, c)), r(__fmul_rn(y0, s))));
            }
          } else if (un.kv == 0) {   // y0' = y0 c - y1 s, y1' = y0 s + y1 c
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float c = cs[16 * rnd + j], s = sn[16 * rnd + j];
              const float y0 = ylo[j], y1 = yhi[j];
              ylo[j] = __fmaf_rn(y0, c, -__fmul_rn(y1, s));
              yhi[j] = __fmaf_rn(y0, s, __fmul_rn(y1, c));
            }
          }
          if (valid) {
#pragma unroll
            for (int v = 0; v < 2; ++v) {
              st_global_hint(out + c_lo + 8 * v,
                             make_uint4(pack_bf16x2(ylo[8 * v], ylo[8 * v + 1]), pack_bf16x2(ylo[8 * v + 2], ylo[8 * v + 3]),
                                        pack_bf16x2(ylo[8 * v + 4], ylo[8 * v + 5]),
                                        pack_bf16x2(ylo[8 * v + 6], ylo[8 * v + 7])),
                             st_pol);
              st_global_hint(out + 64 + c_lo + 8 * v,
                             make_uint4(pack_bf16x2(yhi[8 * v], yhi[8 * v + 1]), pack_bf16x2(yhi[8 * v + 2], yhi[8 * v + 3]),
                                        pack_bf16x2(yhi[8 * v + 4], yhi[8 * v + 5]),
                                        pack_bf16x2(yhi[8 * v + 6], yhi[8 * v + 7])),
                             st_pol);
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  if (warp == 1) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kMTmemCols)
                 : "memory");
  }
}

}  // namespace
}  // namespace kvx

namespace kvx {
namespace {

const char* check_mlp_config(const kvx_mlp_config* c) {
  if (!c) return "NULL config";
  if (c->head_dim != kMD) return "head_dim must be 128";
  if (c->src_layers < 1 || c->tgt_layers < 1 || c->n_kv_heads < 1) return "layer / head counts out of range";
  if (c->k < 1 || c->k > c->src_layers) return "k must be in [1, src_layers]";
  if (c->hidden < 256 || c->hidden % 256 != 0 || c->hidden > 65536) return "hidden must be a multiple of 256";
  if (!(c->src_rope_theta > 1.0) || !(c->tgt_rope_theta > 1.0) || !std::isfinite(c->src_rope_theta) ||
      !std::isfinite(c->tgt_rope_theta))
    return "the RoPE bases must be finite and > 1";
  if (!c->selection) return "NULL selection";
  for (int64_t i = 0; i < static_cast<int64_t>(c->tgt_layers) * c->k; ++i)
    if (c->selection[i] < 0 || c->selection[i] >= c->src_layers) return "selection entry out of range";
  if (!c->W1 || !c->b1 || !c->W2 || !c->b2 || !c->W3 || !c->b3) return "NULL weight or bias";
  const void* ptrs[6] = {c->W1, c->b1, c->W2, c->b2, c->W3, c->b3};
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) & 15u) return "weights and biases must be 16-byte aligned";
  if (static_cast<int64_t>(c->tgt_layers) * 2 * c->n_kv_heads * c->hidden > INT_MAX / 2) return "too many weight rows";
  if (static_cast<int64_t>(c->k) * c->n_kv_heads * kMD > INT_MAX / 2) return "source feature too wide";
  if (c->workspace_bytes != 0 && !c->workspace) return "workspace_bytes without a workspace";
  if (c->rope_numerics != KVX_ROPE_EXACT && c->rope_numerics != KVX_ROPE_HF) return "bad rope_numerics";
  if (const char* why = check_rope_scaling(c->src_rope_scaling)) return why;
  if (const char* why = check_rope_scaling(c->tgt_rope_scaling)) return why;
  if (reinterpret_cast<uintptr_t>(c->workspace) & 255u) return "workspace must be 256-byte aligned";
  return nullptr;
}

size_t al256m(size_t n) { return (n + 255) / 256 * 256; }

// Workspace: stripped source keys, then the two hidden buffers of a group of G target layers.
size_t strip_bytes(const kvx_mlp_config* c, int32_t B, int32_t T) {
  return al256m(static_cast<size_t>(c->src_layers) * B * c->n_kv_heads * T * kMD * 2);
}
size_t hidden_bytes_per_layer(const kvx_mlp_config* c, int32_t B, int32_t T) {
  return static_cast<size_t>(2) * B * T * c->n_kv_heads * c->hidden * 2;   // K and V, bf16
}
// status word and the selection table
size_t table_bytes(const kvx_mlp_config* c) { return al256m(16 + static_cast<size_t>(c->tgt_layers) * c->k * 4); }

}  // namespace
}  // namespace kvx

extern "C" {

KVX_API int64_t kvx_mlp_workspace_bytes(const kvx_mlp_config* cfg, int32_t batch, int32_t tokens_per_seq) {
  using namespace kvx;
  if (check_mlp_config(cfg) || batch < 1 || tokens_per_seq < 1) return -1;
  return static_cast<int64_t>(strip_bytes(cfg, batch, tokens_per_seq) + table_bytes(cfg) +
                              2 * al256m(hidden_bytes_per_layer(cfg, batch, tokens_per_seq) * cfg->tgt_layers));
}

KVX_API kvx_status kvx_mlp_map(const kvx_mlp_config* cfg, const kvx_src* src, int32_t batch, int32_t tokens_per_seq,
                               const int32_t* positions, const kvx_tgt* tgt, void* stream) {
  using namespace kvx;
  NvtxRange range("kvx_mlp_map");
  set_error("");
  auto bad = [](const std::string& m) {
    set_error("kvx_mlp_map: " + m);
    return KVX_ERR_INVALID_ARG;
  };
  if (const char* why = check_mlp_config(cfg)) return bad(why);
  if (!src || !tgt || !positions) return bad("NULL argument");
  if (batch < 0 || tokens_per_seq < 0) return bad("negative batch or tokens_per_seq");
  if (batch == 0 || tokens_per_seq == 0) return KVX_OK;
  if (!src->k || !src->v || !tgt->k || !tgt->v) return bad("NULL cache pointer");
  if (tgt->paged) {
    set_error("kvx_mlp_map: the MLP mapper writes contiguous targets only");
    return KVX_ERR_UNSUPPORTED;
  }
  for (int i = 0; i < 4; ++i)
    if (src->stride[i] < 0 || src->stride[i] % 8 != 0 || tgt->stride[i] < 0 || tgt->stride[i] % 8 != 0)
      return bad("strides must be non-negative multiples of 8");
  if (src->stride[3] < kMD || tgt->stride[3] < kMD) return bad("token stride smaller than head_dim");
  if ((reinterpret_cast<uintptr_t>(src->k) | reinterpret_cast<uintptr_t>(src->v) |
       reinterpret_cast<uintptr_t>(tgt->k) | reinterpret_cast<uintptr_t>(tgt->v)) & 15u)
    return bad("cache pointers must be 16-byte aligned");
  if (reinterpret_cast<uintptr_t>(positions) & 3u) return bad("positions must be 4-byte aligned");
  const int64_t N = static_cast<int64_t>(batch) * tokens_per_seq;
  auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
  if (!encode) {
    set_error("kvx_mlp_map: cuTensorMapEncodeTiled unavailable");
    return KVX_ERR_CUDA;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  int dev = 0, sms = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) {
    set_error(std::string("kvx_mlp_map: device query: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  const int H = cfg->n_kv_heads, Lt = cfg->tgt_layers, hid = cfg->hidden;
  // workspace: stripped keys + status, then H1 / H2 for G target layers at a time
  const size_t sb = strip_bytes(cfg, batch, tokens_per_seq) + table_bytes(cfg);   // strip, status, selection
  const size_t per_layer = hidden_bytes_per_layer(cfg, batch, tokens_per_seq);
  size_t avail = 0;
  char* base = nullptr;
  char* own = nullptr;
  if (cfg->workspace) {
    base = static_cast<char*>(cfg->workspace);
    avail = static_cast<size_t>(cfg->workspace_bytes);
  } else {
    size_t free_b = 0, total_b = 0;
    if ((e = cudaMemGetInfo(&free_b, &total_b)) != cudaSuccess) {
      set_error(std::string("kvx_mlp_map: memory query: ") + cudaGetErrorString(e));
      return KVX_ERR_CUDA;
    }
    avail = std::min<size_t>(free_b / 2, static_cast<size_t>(32) << 30);
    avail = std::min(avail, sb + 2 * al256m(per_layer * Lt));
  }
  if (avail < sb + 2 * al256m(per_layer)) {
    if (cfg->workspace) return bad("workspace too small (see kvx_mlp_workspace_bytes)");
    set_error("kvx_mlp_map: not enough device memory for one target layer's hidden activations");
    return KVX_ERR_OOM;
  }
  // the most target layers whose two hidden buffers fit after the strip and the tables
  int G = static_cast<int>(std::min<size_t>(Lt, (avail - sb) / (2 * per_layer)));
  while (G > 1 && sb + 2 * al256m(per_layer * G) > avail) --G;
  G = std::max(G, 1);
  if (static_cast<int64_t>(G) * 2 * N > INT_MAX - 2 * kMTile) G = static_cast<int>((INT_MAX / 4) / N);
  if (G < 1) return bad("too many tokens for the hidden workspace map");
  if (!cfg->workspace) {
    const size_t need = sb + 2 * al256m(per_layer * G);
    if ((e = cudaMallocAsync(reinterpret_cast<void**>(&own), need, st)) != cudaSuccess) {
      set_error(std::string("kvx_mlp_map: workspace: ") + cudaGetErrorString(e));
      return KVX_ERR_OOM;
    }
    base = own;
  }
  const size_t strip_only = strip_bytes(cfg, batch, tokens_per_seq);
  __nv_bfloat16* d_strip = reinterpret_cast<__nv_bfloat16*>(base);
  int32_t* d_status = reinterpret_cast<int32_t*>(base + strip_only);
  int32_t* d_sel = d_status + 4;
  __nv_bfloat16* d_h1 = reinterpret_cast<__nv_bfloat16*>(base + sb);
  __nv_bfloat16* d_h2 = reinterpret_cast<__nv_bfloat16*>(base + sb + al256m(per_layer * G));
  kvx_status result = KVX_OK;
  do {
    const size_t sel_n = static_cast<size_t>(Lt) * cfg->k;
    if ((e = cudaMemcpyAsync(d_sel, cfg->selection, sel_n * 4, cudaMemcpyHostToDevice, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(d_status, 0, 4, st)) != cudaSuccess) {
      set_error(std::string("kvx_mlp_map: setup: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    kvx_ctx tmp;   // RoPE tables
    tmp.d = kMD;
    tmp.theta_s = cfg->src_rope_theta;
    tmp.theta_t = cfg->tgt_rope_theta;
    set_rope_scaling(&tmp, cfg->src_rope_scaling, cfg->tgt_rope_scaling);
    fill_rope(&tmp);
    MlpParams P;
    std::memset(&P, 0, sizeof(P));
    const cuuint32_t ones[5] = {1, 1, 1, 1, 1};
    auto enc_fail = [&](const char* what) {
      set_error(std::string("kvx_mlp_map: ") + what + " tensor map rejected");
      return KVX_ERR_UNSUPPORTED;
    };
    {
      const cuuint32_t box[5] = {64, kMTile, 1, 1, 1};
      const cuuint64_t dims[5] = {kMD, static_cast<cuuint64_t>(tokens_per_seq), static_cast<cuuint64_t>(H),
                                  static_cast<cuuint64_t>(batch), static_cast<cuuint64_t>(cfg->src_layers)};
      const cuuint64_t row = kMD * 2;
      const cuuint64_t str_ws[4] = {row, row * tokens_per_seq, row * tokens_per_seq * H,
                                    row * tokens_per_seq * H * batch};
      if (encode(&P.tm_ak, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, d_strip, dims, str_ws, box, ones,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
        result = enc_fail("stripped-key");
        break;
      }
      const cuuint64_t str_v[4] = {static_cast<cuuint64_t>(src->stride[3]) * 2, static_cast<cuuint64_t>(src->stride[2]) * 2,
                                   static_cast<cuuint64_t>(src->stride[1]) * 2, static_cast<cuuint64_t>(src->stride[0]) * 2};
      if (encode(&P.tm_av, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(src->v), dims, str_v, box, ones,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
        result = enc_fail("source value");
        break;
      }
    }
    CUtensorMap tm_w1, tm_w2, tm_w3, tm_h1, tm_h2;
    {
      const cuuint32_t box[2] = {64, 128}, box3[2] = {64, 64};
      const int64_t ds = static_cast<int64_t>(cfg->k) * H * kMD;
      const cuuint64_t d1[2] = {static_cast<cuuint64_t>(ds), static_cast<cuuint64_t>(Lt) * 2 * H * hid};
      const cuuint64_t s1[1] = {static_cast<cuuint64_t>(ds) * 2};
      const cuuint64_t d2[2] = {static_cast<cuuint64_t>(hid), static_cast<cuuint64_t>(Lt) * 2 * H * hid};
      const cuuint64_t s2[1] = {static_cast<cuuint64_t>(hid) * 2};
      const cuuint64_t d3[2] = {static_cast<cuuint64_t>(hid), static_cast<cuuint64_t>(Lt) * 2 * H * kMD};
      const cuuint64_t dh[2] = {static_cast<cuuint64_t>(H) * hid, static_cast<cuuint64_t>(G) * 2 * N};
      const cuuint64_t sh[1] = {static_cast<cuuint64_t>(H) * hid * 2};
      if (encode(&tm_w1, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(cfg->W1), d1, s1, box, ones,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
          encode(&tm_w2, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(cfg->W2), d2, s2, box, ones,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
          encode(&tm_w3, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(cfg->W3), d3, s2, box3, ones,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
          encode(&tm_h1, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, d_h1, dh, sh, box, ones, CU_TENSOR_MAP_INTERLEAVE_NONE,
                 CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
          encode(&tm_h2, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, d_h2, dh, sh, box, ones, CU_TENSOR_MAP_INTERLEAVE_NONE,
                 CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
        result = enc_fail("weight or hidden");
        break;
      }
    }
    MapArgs& a = P.a;
    a.src_k = src->k;
    a.src_v = src->v;
    for (int i = 0; i < 4; ++i) {
      a.ss[i] = src->stride[i];
      a.ts[i] = tgt->stride[i];
    }
    a.tgt_k = tgt->k;
    a.tgt_v = tgt->v;
    a.pos = positions;
    a.B = batch;
    a.T = tokens_per_seq;
    P.sel = d_sel;
    P.status = d_status;
    P.H = H;
    P.k = cfg->k;
    P.hidden = hid;
    P.pairs = (tokens_per_seq + 2 * kMTile - 1) / (2 * kMTile);
    P.rope = tmp.rope;
    // strip every source key once
    P.hf = cfg->rope_numerics == KVX_ROPE_HF;
    launch_key_strip(src->k, src->stride, d_strip, positions, cfg->src_layers, H, batch, tokens_per_seq, tmp.rope, sms, st,
                     P.hf, 0);
    const size_t smem = mlp_smem_bytes();
    if ((e = cudaFuncSetAttribute(tc_mlp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem))) != cudaSuccess) {
      set_error(std::string("kvx_mlp_map: smem attribute: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    for (int l0 = 0; l0 < Lt && result == KVX_OK; l0 += G) {
      const int g_n = std::min(G, Lt - l0);
      P.l0 = l0;
      P.G = g_n;
      for (int pass = 1; pass <= 3; ++pass) {
        P.pass = pass;
        P.tm_w = pass == 1 ? tm_w1 : pass == 2 ? tm_w2 : tm_w3;
        P.tm_h = pass == 3 ? tm_h2 : tm_h1;
        P.hout = pass == 1 ? d_h1 : d_h2;
        P.bias = pass == 1 ? cfg->b1 : pass == 2 ? cfg->b2 : cfg->b3;
        P.n_tiles = pass == 1 ? H * hid / 256 : pass == 2 ? hid / 256 : 1;
        P.heads = pass == 1 ? 1 : H;
        P.ksteps = pass == 1 ? cfg->k * H : hid / 128;
        const int64_t units = static_cast<int64_t>(g_n) * 2 * batch * P.pairs * P.heads * P.n_tiles;
        if (units > INT_MAX) {
          set_error("kvx_mlp_map: too many work units");
          result = KVX_ERR_UNSUPPORTED;
          break;
        }
        P.n_units = static_cast<int32_t>(units);
        const int grid = 2 * static_cast<int>(std::min<int64_t>(units, std::max(sms / 2, 1)));
        tc_mlp_kernel<<<grid, kMThreads, smem, st>>>(P);
        if ((e = cudaGetLastError()) != cudaSuccess) {
          set_error(std::string("kvx_mlp_map: launch: ") + cudaGetErrorString(e));
          result = KVX_ERR_CUDA;
          break;
        }
      }
    }
    if (result != KVX_OK) break;
    int32_t dstat = 0;
    if ((e = cudaMemcpyAsync(&dstat, d_status, 4, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess) {
      set_error(std::string("kvx_mlp_map: run: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    if (dstat != 0) {
      set_error(std::string("kvx_mlp_map: device status ") + kvx_status_string(static_cast<kvx_status>(dstat)));
      result = static_cast<kvx_status>(dstat);
    }
  } while (false);
  if (own) cudaFreeAsync(own, st);
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess && result == KVX_OK) {
    set_error(std::string("kvx_mlp_map: ") + cudaGetErrorString(e));
    result = KVX_ERR_CUDA;
  }
  return result;
}

}  // extern "C"
