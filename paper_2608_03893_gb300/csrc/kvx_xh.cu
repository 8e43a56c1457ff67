// Tensor-core path for the cross-head feature layout (the paper's mapper: every KV head of
// the k selected source layers is a feature of every target head, d_s = k n_kv d, Sec. 3.1
// and Sec. 3.2).  bf16 caches and weights, head_dim 128, half-split or interleaved RoPE pairs, an even
// number of KV heads, contiguous or paged targets.  Per-head mappers with more selected
// layers than the per-head kernel holds (k > 4) run here too, on W widened at create time
// with zeros outside each target head's rows.
//
// For target layer l and K|V the map is one GEMM over the tokens,
//   Y[tok][h d + c] = sum_{j, h'} X_{sel[l][j], h'}[tok][:] . W[l][kv][h][(j n_kv + h') d + :][c]
//                     + b[l][kv][h][c],
// then (keys) the target RoPE of each head, as in the per-head kernel (Eq. ridge_kv with
// the Sec. 3.3 composition).  Two kernels:
//
// 1. xh_strip_kernel: the source keys with the source RoPE stripped, rounded to bf16 (the
//    operand rounding of a bf16 forward), written to a workspace [L_s][B][H][T][128].  A
//    thread owns one token and four RoPE pairs and walks every (layer, head), so each
//    cos/sin is computed once per token.  Bound by HBM (read and write of the key cache).
// 2. tc_xh_kernel: clusters of two CTAs; work unit = (target layer, K|V, batch, pair of
//    128-token tiles, pass of two target heads).  The K loop runs over the k n_kv source
//    tiles (layer sel[l][j], head h') in the feature order; each step the CTA pair issues
//    8 pair MMAs (cta_group::2, M = 256, N = 256, K = 16) with A (this CTA's 128 tokens x
//    128 features, straight from the stripped keys or the value cache by TMA) and B (this
//    CTA's 128 of the pass's 256 output rows of W^T) both in shared memory.  Units run
//    pass-fastest and token-tile next, so the clusters in flight share one (layer, K|V)
//    block of W^T (k n_kv d x n_kv d bf16) in L2 and the four passes of a tile share its
//    source tiles.  Epilogue per pass: TMEM -> registers, + bias, (keys) target RoPE,
//    bf16, one TMA store per warp and head (contiguous targets) or 16-byte stores through
//    the block table (paged targets).
//
// Warp roles (384 threads): warp 0 one thread polling two streams (stage loads: A and B
// halves of both CTAs complete on the rank-0 CTA's stage barrier; each unit's bias rows);
// warp 1 TMEM allocator (jointly for the pair) and, in the rank-0 CTA, the MMA issuer;
// warps 4-11 epilogue (thread = one token row x 32 RoPE pairs of each head of the pass).
// Every wait is bounded (KVX_ERR_TIMEOUT, as in the per-head kernel).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <string>
#include <vector>

#include "kvx_internal.h"
#include "kvx_ptx.cuh"
#include "kvx_rope.cuh"
#include "kvx_xh.h"

namespace kvx {
namespace {

using namespace ptx;

constexpr int kXThreads = 384;
constexpr int kXFirstEpi = 4;
constexpr int kXEpiWarps = 8;
constexpr int kXD = 128;                               // head_dim
constexpr int kXTile = 128;                            // tokens per CTA tile
constexpr int kXStages = 3;
constexpr uint32_t kXABytes = kXTile * kXD * 2;        // 32 KB: 128 tokens x 128 features
constexpr uint32_t kXBBytes = 128 * kXD * 2;           // 32 KB: 128 output rows x 128 features
constexpr uint32_t kXStageBytes = kXABytes + kXBBytes;
constexpr uint32_t kXAccCols = 256;                    // two heads x 128 channels, fp32
constexpr uint32_t kXTmemCols = 512;
constexpr uint32_t kXPieceBytes = 32 * 64;             // 32 rows x 32 channels, 64-byte swizzle
constexpr uint32_t kXWarpStage = 2 * kXPieceBytes;     // one warp's share of one head
constexpr int kXBiasSlots = 2;
constexpr uint32_t kXBiasBytes = 2 * kXD * 4;          // the pass's two heads
constexpr size_t kXSmemLimit = 232448;

constexpr size_t xh_smem_bytes() {
  return static_cast<size_t>(kXStages) * kXStageBytes + static_cast<size_t>(kXEpiWarps) * kXWarpStage +
         kXBiasSlots * kXBiasBytes + (2 * kXStages + 4 + 2 * kXBiasSlots + 1) * 8 + 16;
}
static_assert(xh_smem_bytes() <= kXSmemLimit, "cross-head kernel shared memory exceeds the per-CTA limit");

struct XhParams {
  CUtensorMap tm_ak;      // stripped keys [L_s][B][H][T][128] (workspace), box 64 x 128
  CUtensorMap tm_av;      // source values (caller's strides), box 64 x 128
  CUtensorMap tm_w;       // W^T [L_t*2*H*128][F], box 64 x 128
  CUtensorMap tm_out_k;   // targets as (64 ch, T, 2 halves, heads, L_t), box 32 x 32 x 2
  CUtensorMap tm_out_v;
  MapArgs a;
  const int32_t* sel;     // [L_t][k]
  const float* bias;      // [L_t][2][H][128]
  int32_t* status;
  int32_t Lt, H, k, pairs, n_units, out_bh;
  int32_t lo_steps;       // fp32 weights: k n_kv further K steps over the same source tiles with W_lo
  int32_t per_head;       // per-head W widened with zeros: a pass runs only its own two source heads' steps
  int32_t hf;             // the Hugging Face forward's RoPE rounding (kvx_rope_numerics)
  int32_t il;             // interleaved RoPE pairs (2i, 2i+1) instead of (i, i + 64)
  RopeTables rope;
};

struct XUnit {
  int l, kv, b, t0, pass;
};

// Unit order: pass fastest, then tile pair, batch, K|V, target layer (see the header).
__device__ __forceinline__ XUnit xh_decode(int u, int H, int B, int pairs, uint32_t rank) {
  XUnit r;
  const int passes = H / 2;
  r.pass = u % passes;
  int rest = u / passes;
  r.t0 = (2 * (rest % pairs) + static_cast<int>(rank)) * kXTile;
  rest /= pairs;
  r.b = rest % B;
  rest /= B;
  r.kv = rest % 2;
  r.l = rest / 2;
  return r;
}

__device__ __forceinline__ void xreport(int32_t* status, int code) { atomicCAS(status, 0, code); }

// ---------------------------------------------------------------- strip kernel --
// Thread = (sequence b, token t, group of four RoPE pairs i0..i0+3); it rotates those
// pairs of every (source layer, head) by -t*omega_s and rounds them to bf16.  Half-split
// pairs (i, i + 64) take channels 4 grp .. 4 grp + 3 and 64 + the same; interleaved pairs
// (2i, 2i+1) take channels 8 grp .. 8 grp + 7.
__global__ void __launch_bounds__(256) xh_strip_kernel(const __nv_bfloat16* __restrict__ src, int64_t s_l,
                                                       int64_t s_b, int64_t s_h, int64_t s_t,
                                                       __nv_bfloat16* __restrict__ ws, const int32_t* __restrict__ pos,
                                                       int Ls, int H, int B, int T, RopeTables rope, int hf, int il) {
  const int64_t n = static_cast<int64_t>(B) * T * 16;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int grp = static_cast<int>(i % 16);
    const int64_t bt = i / 16;
    const int t = static_cast<int>(bt % T), b = static_cast<int>(bt / T);
    int p = __ldg(&pos[bt]);
    if (p < 0 || p >= (1 << 24)) p = 0;   // the mapping kernel reports the position
    float c[4], s[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      if (hf) {   // HF numerics: cos / sin of the fp32 angle, rounded to bf16
        sincosf(__fmul_rn(static_cast<float>(p), rope.ws_hi[4 * grp + m]), &s[m], &c[m]);
        s[m] = __bfloat162float(__float2bfloat16_rn(s[m]));
        c[m] = __bfloat162float(__float2bfloat16_rn(c[m]));
      } else {
        rope_sincos(p, rope.ws_hi[4 * grp + m], rope.ws_lo[4 * grp + m], rope.two_pi_hi, rope.two_pi_lo,
                    rope.inv_two_pi, &s[m], &c[m]);
      }
    }
    for (int L = 0; L < Ls; ++L) {
      for (int h = 0; h < H; ++h) {
        const __nv_bfloat16* row = src + L * s_l + b * s_b + h * s_h + static_cast<int64_t>(t) * s_t;
        uint4 vi;
        if (il) {
          vi = *reinterpret_cast<const uint4*>(row + 8 * grp);
        } else {
          const uint2 va = *reinterpret_cast<const uint2*>(row + 4 * grp);        // first halves
          const uint2 vb = *reinterpret_cast<const uint2*>(row + 64 + 4 * grp);   // second halves
          vi = make_uint4(va.x, vb.x, va.y, vb.y);
        }
        uint32_t oa[2], ob[2];
#pragma unroll
        for (int w = 0; w < 2; ++w) {
          // half-split: vi = (a01, b01, a23, b23) with a = first members; interleaved: vi
          // = (pair 0, pair 1, pair 2, pair 3), one pair per word
          const uint32_t u0 = w ? vi.z : vi.x, u1 = w ? vi.w : vi.y;
          float a0, a1, b0, b1;
          if (il) {
            a0 = bf16_lo(u0); b0 = bf16_hi(u0); a1 = bf16_lo(u1); b1 = bf16_hi(u1);
          } else {
            a0 = bf16_lo(u0); a1 = bf16_hi(u0); b0 = bf16_lo(u1); b1 = bf16_hi(u1);
          }
          const int m0 = 2 * w, m1 = 2 * w + 1;
          float na0, na1, nb0, nb1;
          if (hf) {   // each product and sum rounded to bf16
            auto r = [](float x) { return __bfloat162float(__float2bfloat16_rn(x)); };
            na0 = r(__fadd_rn(r(__fmul_rn(a0, c[m0])), r(__fmul_rn(b0, s[m0]))));
            na1 = r(__fadd_rn(r(__fmul_rn(a1, c[m1])), r(__fmul_rn(b1, s[m1]))));
            nb0 = r(__fsub_rn(r(__fmul_rn(b0, c[m0])), r(__fmul_rn(a0, s[m0]))));
            nb1 = r(__fsub_rn(r(__fmul_rn(b1, c[m1])), r(__fmul_rn(a1, s[m1]))));
          } else {
            // rotation by -t*omega: a' = a c + b s, b' = b c - a s
            na0 = __fmaf_rn(a0, c[m0], __fmul_rn(b0, s[m0]));
            na1 = __fmaf_rn(a1, c[m1], __fmul_rn(b1, s[m1]));
            nb0 = __fmaf_rn(b0, c[m0], -__fmul_rn(a0, s[m0]));
            nb1 = __fmaf_rn(b1, c[m1], -__fmul_rn(a1, s[m1]));
          }
          if (il) {
            oa[w] = pack_bf16x2(na0, nb0);
            ob[w] = pack_bf16x2(na1, nb1);
          } else {
            oa[w] = pack_bf16x2(na0, na1);
            ob[w] = pack_bf16x2(nb0, nb1);
          }
        }
        __nv_bfloat16* out = ws + ((((static_cast<int64_t>(L) * B + b) * H + h) * T + t) * kXD);
        if (il) {
          *reinterpret_cast<uint4*>(out + 8 * grp) = make_uint4(oa[0], ob[0], oa[1], ob[1]);
        } else {
          *reinterpret_cast<uint2*>(out + 4 * grp) = make_uint2(oa[0], oa[1]);
          *reinterpret_cast<uint2*>(out + 64 + 4 * grp) = make_uint2(ob[0], ob[1]);
        }
      }
    }
  }
}

// -------------------------------------------------------------- mapping kernel --

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kXThreads, 1)
    tc_xh_kernel(const __grid_constant__ XhParams P) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) xreport(P.status, KVX_ERR_UNSUPPORTED);
    return;
  }
  uint8_t* stages = smem;                                          // [3] x (A 32 KB | B 32 KB)
  uint8_t* outst = stages + static_cast<size_t>(kXStages) * kXStageBytes;
  float* bias_ring = reinterpret_cast<float*>(outst + kXEpiWarps * kXWarpStage);   // [2][256]
  uint64_t* bars = reinterpret_cast<uint64_t*>(bias_ring + kXBiasSlots * 2 * kXD);
  uint64_t* full = bars;                          // [3] both CTAs' A and B landed (rank 0)
  uint64_t* empty = full + kXStages;              // [3] the stage's MMAs completed
  uint64_t* accf = empty + kXStages;              // [2] accumulator ready
  uint64_t* acce = accf + 2;                      // [2] accumulator drained (8 warps x 2 CTAs, rank 0)
  uint64_t* bias_full = acce + 2;                 // [2]
  uint64_t* bias_empty = bias_full + kXBiasSlots; // [2] (8 epilogue warps)
  uint64_t* drain = bias_empty + kXBiasSlots;     // [1]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  volatile uint32_t* abort_flag = tmem_holder + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int unit0 = blockIdx.x >> 1, unit_step = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kXStages; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accf[i]), 1);
      mbar_init(smem_u32(&acce[i]), 2 * kXEpiWarps);
    }
    for (int i = 0; i < kXBiasSlots; ++i) {
      mbar_init(smem_u32(&bias_full[i]), 1);
      mbar_init(smem_u32(&bias_empty[i]), kXEpiWarps);
    }
    mbar_init(smem_u32(&drain[0]), 1);
    *abort_flag = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(kXTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // A unit's K steps: (layer j, head hs) source tiles in the feature order, then (fp32 W) the
  // same again with W_lo.  For a per-head mapper (W widened with zeros outside each head's
  // rows) only the pass's own heads hs = 2 pass, 2 pass + 1 meet non-zero rows, so the unit
  // runs those 2k steps alone.
  const int H = P.H, k = P.k, src_steps = P.k * P.H;
  const int unit_src = P.per_head ? 2 * P.k : src_steps;
  const int steps = unit_src * (P.lo_steps ? 2 : 1);
  const int n_units = P.n_units, pairs = P.pairs;
  const MapArgs& A = P.a;

  if (warp == 0) {
    // -------------------------------------------------- stage and bias producer ------
    if (lane == 0) {
      const uint64_t pol_a = policy_evict_first();
      const uint64_t pol_w = policy_evict_last();
      uint32_t sn = 0, bn = 0;
      int su = unit0, ss = 0, bu = unit0;
      XUnit sun = xh_decode(su < n_units ? su : 0, H, A.B, pairs, rank);
      bool ok = true;
      uint64_t t_idle = 0;
      uint32_t spins = 0;
      for (;;) {
        bool busy = false, progress = false;
        if (su < n_units) {
          busy = true;
          const int st = static_cast<int>(sn % kXStages);
          const uint32_t round = sn / kXStages;
          if (round == 0 || mbar_test_wait(smem_u32(&empty[st]), (round - 1) & 1u)) {
            // step ss -> feature block fb: source layer sel[l][(fb % src_steps) / H], head
            // fb % H; W^T columns fb*128 ..
            int fb = ss;
            if (P.per_head) {
              const int part = ss / unit_src, s2 = ss % unit_src;
              fb = part * src_steps + (s2 >> 1) * H + 2 * sun.pass + (s2 & 1);
            }
            const int j = (fb % src_steps) / H, hs = fb % H;
            const int L = __ldg(&P.sel[sun.l * k + j]);
            if (rank == 0) mbar_expect_tx(smem_u32(&full[st]), 2 * kXStageBytes);
            const uint32_t bar = mapa_shared(smem_u32(&full[st]), 0);
            const uint32_t a_dst = smem_u32(stages + static_cast<size_t>(st) * kXStageBytes);
            const uint32_t b_dst = a_dst + kXABytes;
            const CUtensorMap* tma = sun.kv ? &P.tm_av : &P.tm_ak;
            tma_load_5d_pair(a_dst, tma, bar, 0, sun.t0, hs, sun.b, L, pol_a);
            tma_load_5d_pair(a_dst + kXABytes / 2, tma, bar, 64, sun.t0, hs, sun.b, L, pol_a);
            const int wrow = ((sun.l * 2 + sun.kv) * H + 2 * sun.pass) * kXD + static_cast<int>(rank) * 128;
            tma_load_2d_pair(b_dst, &P.tm_w, bar, fb * kXD, wrow, pol_w);
            tma_load_2d_pair(b_dst + kXBBytes / 2, &P.tm_w, bar, fb * kXD + 64, wrow, pol_w);
            ++sn;
            if (++ss == steps) {
              ss = 0;
              su += unit_step;
              if (su < n_units) sun = xh_decode(su, H, A.B, pairs, rank);
            }
            progress = true;
          }
        }
        if (bu < n_units) {
          busy = true;
          const int bs = static_cast<int>(bn % kXBiasSlots);
          const uint32_t round = bn / kXBiasSlots;
          if (round == 0 || mbar_test_wait(smem_u32(&bias_empty[bs]), (round - 1) & 1u)) {
            const XUnit bun = xh_decode(bu, H, A.B, pairs, rank);
            const int row0 = ((bun.l * 2 + bun.kv) * H + 2 * bun.pass) * kXD;
            mbar_expect_tx(smem_u32(&bias_full[bs]), kXBiasBytes);
            bulk_load(smem_u32(bias_ring + bs * 2 * kXD), P.bias + static_cast<size_t>(row0), kXBiasBytes,
                      smem_u32(&bias_full[bs]));
            ++bn;
            bu += unit_step;
            progress = true;
          }
        }
        if (!busy) break;
        if (progress) {
          spins = 0;
          t_idle = 0;
          continue;
        }
        if ((++spins & 63u) == 0) {   // bounded: no slot freed for 4 s raises KVX_ERR_TIMEOUT
          if (*abort_flag) {
            ok = false;
            break;
          }
          const uint64_t now = global_timer();
          if (t_idle == 0) {
            t_idle = now;
          } else if (now - t_idle > kTimeoutNs) {
            *abort_flag = 1u;
            xreport(P.status, KVX_ERR_TIMEOUT);
            ok = false;
            break;
          }
        }
      }
      if (!ok) {   // the most recent loads may still be landing
        if (rank == 0) {
          const uint32_t first = sn > static_cast<uint32_t>(kXStages) ? sn - kXStages : 0;
          for (uint32_t i = first; i < sn; ++i) drain_wait(smem_u32(&full[i % kXStages]), (i / kXStages) & 1u);
        }
        const uint32_t bfirst = bn > static_cast<uint32_t>(kXBiasSlots) ? bn - kXBiasSlots : 0;
        for (uint32_t i = bfirst; i < bn; ++i)
          drain_wait(smem_u32(&bias_full[i % kXBiasSlots]), (i / kXBiasSlots) & 1u);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issuer ------
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = make_idesc(2 * kXTile, 256);   // M = 256 (both CTAs), N = 256
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
        const uint32_t d_tmem = tmem_base + buf * kXAccCols;
        for (int s = 0; s < steps; ++s, ++si) {
          const uint32_t st = si % kXStages;
          if (!wait_bar(smem_u32(&full[st]), (si / kXStages) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(stages + static_cast<size_t>(st) * kXStageBytes);
          const uint32_t b0 = a0 + kXABytes;
#pragma unroll
          for (int half = 0; half < 2; ++half)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_ss_pair(d_tmem, sw128_desc(a0 + half * (kXABytes / 2) + kk * 32),
                             sw128_desc(b0 + half * (kXBBytes / 2) + kk * 32), idesc, (s | half | kk) != 0);
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
  } else if (warp >= kXFirstEpi) {
    // -------------------------------------------------------------- epilogue ------
    const int g = (warp - kXFirstEpi) >> 2;          // pairs 32g .. 32g+31 of each head
    const int q = warp & 3;                          // TMEM lane quarter
    const int r = q * 32 + lane;                     // token row within the tile
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    const uint64_t st_pol = policy_evict_first();
    uint32_t acc_n = 0, bn = 0, stores = 0;
    uint8_t* sb = outst + static_cast<size_t>(warp - kXFirstEpi) * kXWarpStage;
    float cs[32], sn[32];
    bool ok = true;
    for (int u = unit0; ok && u < n_units; u += unit_step, ++acc_n, ++bn) {
      const XUnit un = xh_decode(u, H, A.B, pairs, rank);
      const int t = un.t0 + r;
      bool valid = t < A.T;
      bool bad = false;
      int p = 0;
      if (valid) {
        p = __ldg(&A.pos[static_cast<int64_t>(un.b) * A.T + t]);
        if (p < 0 || p >= (1 << 24)) {
          xreport(P.status, KVX_ERR_DEVICE_BOUNDS);
          valid = false;
          bad = true;
          p = 0;
        }
      }
      // the row's element offset within a target layer, without the head term: contiguous
      // (batch, token) or paged (block through the block table, slot)
      int64_t row_off = 0;
      if (valid) {
        if (!A.paged) {
          row_off = un.b * A.ts[1] + static_cast<int64_t>(t) * A.ts[3];
        } else {
          const int lb = p / A.block_size;
          const int blk =
              lb < A.max_blocks ? __ldg(&A.block_table[static_cast<int64_t>(un.b) * A.max_blocks + lb]) : -1;
          if (blk < 0 || blk >= A.n_blocks) {
            xreport(P.status, KVX_ERR_DEVICE_BOUNDS);
            valid = false;
          } else {
            row_off = static_cast<int64_t>(blk) * A.ts[1] + static_cast<int64_t>(p % A.block_size) * A.ts[3];
          }
        }
      }
      const bool warp_tma = P.out_bh != 0 && __ballot_sync(0xffffffffu, bad) == 0u;
      if (un.kv == 0) {
#pragma unroll
        for (int m = 0; m < 32; ++m) {
          // pair of slot m: half-split pairs (c, c + 64) for c = 32g + m; interleaved pairs
          // (c, c + 1) for the 16 even c in [32g, 32g + 32) (m < 16), then in 64 + [32g, 32g + 32)
          const int i = P.il ? (m < 16 ? 16 * g + m : 32 + 16 * g + (m - 16)) : 32 * g + m;
          if (P.hf) {   // cos / sin of the fp32 angle, rounded to bf16
            sincosf(__fmul_rn(static_cast<float>(p), P.rope.wt_hi[i]), &sn[m], &cs[m]);
            sn[m] = bf16_round(sn[m]);
            cs[m] = bf16_round(cs[m]);
          } else {
            rope_sincos(p, P.rope.wt_hi[i], P.rope.wt_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi,
                        &sn[m], &cs[m]);
          }
        }
      }
      const uint32_t bslot = bn % kXBiasSlots;
      const uint32_t buf = acc_n & 1u;
      bool w_ok = wait_bar(smem_u32(&bias_full[bslot]), (bn / kXBiasSlots) & 1u, abort_flag, P.status,
                           KVX_ERR_TIMEOUT);
      w_ok = w_ok && wait_bar(smem_u32(&accf[buf]), (acc_n >> 1) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT);
      if (!__all_sync(0xffffffffu, w_ok)) {
        ok = false;
        break;
      }
      tc_fence_after();
      __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(un.kv ? A.tgt_v : A.tgt_k);
      const CUtensorMap* tm_out = un.kv ? &P.tm_out_v : &P.tm_out_k;
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        const int h = 2 * un.pass + hh;
        const float* bias = bias_ring + bslot * 2 * kXD + hh * kXD;
        // the staging buffer is free once this warp's previous store has read it
        if (stores > 0) {
          if (lane == 0) bulk_wait_read_all();
          __syncwarp();
        }
        const uint32_t col = tmem_base + lane_addr + buf * kXAccCols + hh * kXD + 32 * g;
#pragma unroll
        for (int rnd = 0; rnd < 2; ++rnd) {
          uint32_t lo[16], hi[16];
          tmem_ld_2x16(col + 16 * rnd, col + 64 + 16 * rnd, lo, hi);
          if (hh == 1 && rnd == 1) {   // the accumulator is free for the unit after next
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&acce[buf]), 0));
          }
          const int c_lo = 32 * g + 16 * rnd;   // channels c_lo + [0,16) and 64 + c_lo + [0,16)
          float ylo[16], yhi[16];
#pragma unroll
          for (int j = 0; j < 16; j += 4) {
            const float4 b0 = *reinterpret_cast<const float4*>(bias + c_lo + j);
            const float4 b1 = *reinterpret_cast<const float4*>(bias + 64 + c_lo + j);
            ylo[j] = __fadd_rn(__uint_as_float(lo[j]), b0.x);
            ylo[j + 1] = __fadd_rn(__uint_as_float(lo[j + 1]), b0.y);
            ylo[j + 2] = __fadd_rn(__uint_as_float(lo[j + 2]), b0.z);
            ylo[j + 3] = __fadd_rn(__uint_as_float(lo[j + 3]), b0.w);
            yhi[j] = __fadd_rn(__uint_as_float(hi[j]), b1.x);
            yhi[j + 1] = __fadd_rn(__uint_as_float(hi[j + 1]), b1.y);
            yhi[j + 2] = __fadd_rn(__uint_as_float(hi[j + 2]), b1.z);
            yhi[j + 3] = __fadd_rn(__uint_as_float(hi[j + 3]), b1.w);
          }
          // target RoPE, two pairs per f32x2 instruction: y0' = y0 c - y1 s, y1' = y0 s + y1 c;
          // HF numerics: the key as bf16, products and sums rounded to bf16
          auto rot = [&](float2 y0, float2 y1, float2 c, float2 sv, float2& r0, float2& r1) {
            if (P.hf) {
              const float2 b0 = bf16_round2(y0), b1 = bf16_round2(y1);
              const float2 p0 = bf16_round2(__fmul2_rn(b0, c)), p1 = bf16_round2(__fmul2_rn(b1, sv));
              const float2 p2 = bf16_round2(__fmul2_rn(b1, c)), p3 = bf16_round2(__fmul2_rn(b0, sv));
              r0 = make_float2(__fsub_rn(p0.x, p1.x), __fsub_rn(p0.y, p1.y));
              r1 = make_float2(__fadd_rn(p2.x, p3.x), __fadd_rn(p2.y, p3.y));
            } else {
              const float2 uu = __fmul2_rn(y1, sv);
              r0 = __ffma2_rn(y0, c, make_float2(-uu.x, -uu.y));
              r1 = __ffma2_rn(y0, sv, __fmul2_rn(y1, c));
            }
          };
          if (un.kv == 0 && !P.il) {   // pairs (c, c + 64): channel c_lo + j of ylo with the same of yhi
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
              float2 r0, r1;
              rot(make_float2(ylo[j], ylo[j + 1]), make_float2(yhi[j], yhi[j + 1]),
                  make_float2(cs[16 * rnd + j], cs[16 * rnd + j + 1]), make_float2(sn[16 * rnd + j], sn[16 * rnd + j + 1]),
                  r0, r1);
              ylo[j] = r0.x;
              ylo[j + 1] = r0.y;
              yhi[j] = r1.x;
              yhi[j + 1] = r1.y;
            }
          } else if (un.kv == 0) {
            // pairs (c, c + 1): channels c_lo + j, c_lo + j + 1 of ylo (slot 8 rnd + j / 2) and
            // of yhi (slot 16 + 8 rnd + j / 2)
#pragma unroll
            for (int j = 0; j < 16; j += 4) {
              const int m = 8 * rnd + j / 2;
              float2 r0, r1;
              rot(make_float2(ylo[j], ylo[j + 2]), make_float2(ylo[j + 1], ylo[j + 3]), make_float2(cs[m], cs[m + 1]),
                  make_float2(sn[m], sn[m + 1]), r0, r1);
              ylo[j] = r0.x;
              ylo[j + 2] = r0.y;
              ylo[j + 1] = r1.x;
              ylo[j + 3] = r1.y;
              rot(make_float2(yhi[j], yhi[j + 2]), make_float2(yhi[j + 1], yhi[j + 3]),
                  make_float2(cs[16 + m], cs[17 + m]), make_float2(sn[16 + m], sn[17 + m]), r0, r1);
              yhi[j] = r0.x;
              yhi[j + 2] = r0.y;
              yhi[j + 1] = r1.x;
              yhi[j + 3] = r1.y;
            }
          }
          uint4 v[4];
          v[0] = make_uint4(pack_bf16x2(ylo[0], ylo[1]), pack_bf16x2(ylo[2], ylo[3]), pack_bf16x2(ylo[4], ylo[5]),
                            pack_bf16x2(ylo[6], ylo[7]));
          v[1] = make_uint4(pack_bf16x2(ylo[8], ylo[9]), pack_bf16x2(ylo[10], ylo[11]),
                            pack_bf16x2(ylo[12], ylo[13]), pack_bf16x2(ylo[14], ylo[15]));
          v[2] = make_uint4(pack_bf16x2(yhi[0], yhi[1]), pack_bf16x2(yhi[2], yhi[3]), pack_bf16x2(yhi[4], yhi[5]),
                            pack_bf16x2(yhi[6], yhi[7]));
          v[3] = make_uint4(pack_bf16x2(yhi[8], yhi[9]), pack_bf16x2(yhi[10], yhi[11]),
                            pack_bf16x2(yhi[12], yhi[13]), pack_bf16x2(yhi[14], yhi[15]));
          if (warp_tma) {
            // two 32-row x 64-byte pieces (channels 32g.. and 64+32g..), 64-byte swizzle:
            // 16-byte chunk index XOR (row / 2) % 4
            const int sw = (lane >> 1) & 3;
            uint8_t* prow = sb + lane * 64;
            *reinterpret_cast<uint4*>(prow + (((2 * rnd) ^ sw) << 4)) = v[0];
            *reinterpret_cast<uint4*>(prow + (((2 * rnd + 1) ^ sw) << 4)) = v[1];
            *reinterpret_cast<uint4*>(prow + kXPieceBytes + (((2 * rnd) ^ sw) << 4)) = v[2];
            *reinterpret_cast<uint4*>(prow + kXPieceBytes + (((2 * rnd + 1) ^ sw) << 4)) = v[3];
          } else if (valid) {
            __nv_bfloat16* out = dst + static_cast<int64_t>(un.l) * A.ts[0] + row_off + static_cast<int64_t>(h) * A.ts[2];
            st_global_hint(out + c_lo, v[0], st_pol);
            st_global_hint(out + c_lo + 8, v[1], st_pol);
            st_global_hint(out + 64 + c_lo, v[2], st_pol);
            st_global_hint(out + 64 + c_lo + 8, v[3], st_pol);
          }
        }
        // every head commits one bulk group per warp (empty when the rows went out directly)
        if (warp_tma) fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (warp_tma && un.t0 + 32 * q < A.T) {   // skip a box wholly past the sequence end
            const int bh = P.out_bh == 2 ? un.b * H + h : h;
            tma_store_5d(tm_out, smem_u32(sb), 32 * g, un.t0 + 32 * q, 0, bh, un.l);
          }
          bulk_commit_group();
        }
        ++stores;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bias_empty[bslot]));
    }
    if (lane == 0) bulk_wait_all();   // this warp's stores are complete
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  if (warp == 1) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kXTmemCols)
                 : "memory");
  }
}

}  // namespace

kvx_status repack_wt_hilo(kvx_ctx* c, const void* W_host, size_t F) {
  // W fp32 [L_t][2][H][F][128] -> W^T bf16 [L_t][2][H][128][2F]: columns [0, F) hold
  // hi = bf16(w), columns [F, 2F) lo = bf16(w - hi), so X W = X W_hi + X W_lo to within
  // 2^-17 of each weight (the paper keeps W in fp32)
  const size_t blocks = static_cast<size_t>(c->Lt) * 2 * c->H;
  std::vector<uint16_t> wt(blocks * 2 * F * kXD);
  const float* w = static_cast<const float*>(W_host);
  auto bf16_rne = [](float x, float* back) {
    uint32_t u;
    std::memcpy(&u, &x, 4);
    if ((u & 0x7F800000u) != 0x7F800000u) u += 0x7FFFu + ((u >> 16) & 1u);   // round to nearest even
    const uint32_t r = u & 0xFFFF0000u;
    std::memcpy(back, &r, 4);
    return static_cast<uint16_t>(r >> 16);
  };
  for (size_t blk = 0; blk < blocks; ++blk) {
    const float* srcb = w + blk * F * kXD;
    uint16_t* dstb = wt.data() + blk * 2 * F * kXD;
    for (size_t f = 0; f < F; ++f)
      for (int n = 0; n < kXD; ++n) {
        const float x = srcb[f * kXD + n];
        float hi = 0.f, lo = 0.f;
        const uint16_t h = bf16_rne(x, &hi);
        const uint16_t l = bf16_rne(x - hi, &lo);
        dstb[static_cast<size_t>(n) * 2 * F + f] = h;
        dstb[static_cast<size_t>(n) * 2 * F + F + f] = l;
      }
  }
  cudaError_t e = cudaMalloc(&c->d_Wt, wt.size() * 2);
  if (e != cudaSuccess) {
    set_error(std::string("kvx_create: cudaMalloc W^T: ") + cudaGetErrorString(e));
    return KVX_ERR_OOM;
  }
  if ((e = cudaMemcpy(c->d_Wt, wt.data(), wt.size() * 2, cudaMemcpyHostToDevice)) != cudaSuccess) {
    set_error(std::string("kvx_create: upload W^T: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

void launch_key_strip(const void* src_k, const int64_t* ss, void* ws, const int32_t* pos, int Ls, int H, int B, int T,
                      const RopeTables& rope, int sms, cudaStream_t stream, int hf, int il) {
  const int64_t threads = static_cast<int64_t>(B) * T * 16;
  const int blocks = static_cast<int>(std::min<int64_t>((threads + 255) / 256, static_cast<int64_t>(sms) * 8));
  xh_strip_kernel<<<blocks, 256, 0, stream>>>(static_cast<const __nv_bfloat16*>(src_k), ss[0], ss[1], ss[2], ss[3],
                                              static_cast<__nv_bfloat16*>(ws), pos, Ls, H, B, T, rope, hf, il);
}

bool xh_supported(const kvx_ctx* c, std::string* why) {
  std::string w;
  if (c->cache_dtype != KVX_BF16) w = "needs bf16 caches";
  else if (c->d != kXD) w = "needs head_dim 128";
  else if (c->head_mix != KVX_CROSS_HEAD && c->k <= 4)
    w = "runs per-head mappers only for k > 4 (the per-head tensor-core kernel takes k <= 4)";
  else if (c->H % 2 != 0) w = "needs an even number of KV heads";
  else if (static_cast<int64_t>(c->Lt) * 2 * c->H * kXD > INT_MAX ||
           static_cast<int64_t>(c->k) * c->H * kXD > INT_MAX / 2)
    w = "too many W rows";
  if (why) *why = w;
  return w.empty();
}

kvx_status launch_xh(kvx_ctx* c, const MapArgs& a, cudaStream_t stream) {
  auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
  if (!encode) {
    set_error("kvx_map: cuTensorMapEncodeTiled unavailable");
    return KVX_ERR_CUDA;
  }
  // workspace for the stripped keys, kept by the context and grown on demand
  const size_t ws_bytes = static_cast<size_t>(c->Ls) * a.B * c->H * a.T * kXD * 2;
  cudaError_t e;
  if (c->ws_bytes < ws_bytes) {
    cudaFree(c->d_ws);
    c->d_ws = nullptr;
    c->ws_bytes = 0;
    if ((e = cudaMalloc(&c->d_ws, ws_bytes)) != cudaSuccess) {
      set_error(std::string("kvx_map: cudaMalloc cross-head workspace: ") + cudaGetErrorString(e));
      return KVX_ERR_OOM;
    }
    c->ws_bytes = ws_bytes;
  }
  XhParams P;
  std::memset(&P, 0, sizeof(P));
  const cuuint32_t ones[5] = {1, 1, 1, 1, 1};
  const cuuint32_t box[5] = {64, kXTile, 1, 1, 1};
  {  // stripped keys: the workspace, contiguous [L_s][B][H][T][128]
    const cuuint64_t dims[5] = {static_cast<cuuint64_t>(kXD), static_cast<cuuint64_t>(a.T),
                                static_cast<cuuint64_t>(c->H), static_cast<cuuint64_t>(a.B),
                                static_cast<cuuint64_t>(c->Ls)};
    const cuuint64_t row = static_cast<cuuint64_t>(kXD) * 2;
    const cuuint64_t str[4] = {row, row * a.T, row * a.T * c->H, row * a.T * c->H * a.B};
    CUresult r = encode(&P.tm_ak, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, c->d_ws, dims, str, box, ones,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      set_error("kvx_map: workspace tensor map rejected");
      return KVX_ERR_UNSUPPORTED;
    }
  }
  {  // source values with the caller's strides
    const cuuint64_t dims[5] = {static_cast<cuuint64_t>(kXD), static_cast<cuuint64_t>(a.T),
                                static_cast<cuuint64_t>(c->H), static_cast<cuuint64_t>(a.B),
                                static_cast<cuuint64_t>(c->Ls)};
    const cuuint64_t str[4] = {static_cast<cuuint64_t>(a.ss[3]) * 2, static_cast<cuuint64_t>(a.ss[2]) * 2,
                               static_cast<cuuint64_t>(a.ss[1]) * 2, static_cast<cuuint64_t>(a.ss[0]) * 2};
    CUresult r = encode(&P.tm_av, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(a.src_v), dims, str, box,
                        ones, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      set_error("kvx_map: source tensor map rejected (strides or sizes)");
      return KVX_ERR_UNSUPPORTED;
    }
  }
  // targets: as in the per-head kernel, (64 channels, T, 2 halves, heads, L_t), box 32 x 32 x 2;
  // paged targets take 16-byte stores through the block table
  P.out_bh = 0;
  if (!a.paged && (a.B == 1 || a.ts[1] == static_cast<int64_t>(c->H) * a.ts[2])) {
    P.out_bh = a.B == 1 ? 1 : 2;
    const cuuint32_t tbox[5] = {32, 32, 2, 1, 1};
    const cuuint64_t tdims[5] = {64, static_cast<cuuint64_t>(a.T), 2,
                                 static_cast<cuuint64_t>(c->H) * static_cast<cuuint64_t>(a.B),
                                 static_cast<cuuint64_t>(c->Lt)};
    const cuuint64_t tstr[4] = {static_cast<cuuint64_t>(a.ts[3]) * 2, 64 * 2, static_cast<cuuint64_t>(a.ts[2]) * 2,
                                static_cast<cuuint64_t>(a.ts[0]) * 2};
    for (int kv = 0; kv < 2; ++kv) {
      CUresult r = encode(kv ? &P.tm_out_v : &P.tm_out_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                          kv ? a.tgt_v : a.tgt_k, tdims, tstr, tbox, ones, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS) {
        set_error("kvx_map: target tensor map rejected (strides or sizes)");
        return KVX_ERR_UNSUPPORTED;
      }
    }
  }
  {  // W^T [L_t*2*H*128][F], box 64 features x 128 rows
    // fp32 weights: W^T holds [W_hi | W_lo], 2F columns (see repack_wt_hilo)
    const cuuint64_t wcols = static_cast<cuuint64_t>(c->F_xh) * (c->weight_dtype == KVX_F32 ? 2 : 1);
    const cuuint64_t wdims[2] = {wcols, static_cast<cuuint64_t>(c->Lt) * 2 * c->H * kXD};
    const cuuint64_t wstr[1] = {wcols * 2};
    const cuuint32_t wbox[2] = {64, 128};
    CUresult r = encode(&P.tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->d_Wt, wdims, wstr, wbox, ones,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      set_error("kvx_map: weight tensor map rejected");
      return KVX_ERR_CUDA;
    }
  }
  P.a = a;
  P.sel = c->d_sel;
  P.bias = c->d_b;
  P.status = c->d_status;
  P.Lt = c->Lt;
  P.H = c->H;
  P.k = c->k;
  P.pairs = (a.T + 2 * kXTile - 1) / (2 * kXTile);
  const int64_t units = static_cast<int64_t>(c->Lt) * 2 * a.B * P.pairs * (c->H / 2);
  if (units > INT_MAX) {
    set_error("kvx_map: too many work units");
    return KVX_ERR_UNSUPPORTED;
  }
  P.n_units = static_cast<int>(units);
  P.lo_steps = c->weight_dtype == KVX_F32 ? c->k * c->H : 0;
  P.per_head = c->head_mix == KVX_PER_HEAD ? 1 : 0;
  P.hf = c->rope_numerics == KVX_ROPE_HF;
  P.il = c->rope_style == KVX_ROPE_INTERLEAVED;
  P.rope = c->rope;

  // 1. strip the source RoPE from every key into the workspace
  {
    launch_key_strip(a.src_k, a.ss, c->d_ws, a.pos, c->Ls, c->H, a.B, a.T, c->rope, c->sm_count, stream,
                     c->rope_numerics == KVX_ROPE_HF, c->rope_style == KVX_ROPE_INTERLEAVED);
    if ((e = cudaGetLastError()) != cudaSuccess) {
      set_error(std::string("kvx_map: strip launch: ") + cudaGetErrorString(e));
      return KVX_ERR_CUDA;
    }
  }
  // 2. the GEMMs
  const size_t smem = xh_smem_bytes();
  if ((e = cudaFuncSetAttribute(tc_xh_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem))) != cudaSuccess) {
    set_error(std::string("kvx_map: smem attribute: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  const int grid = 2 * static_cast<int>(std::min<int64_t>(units, std::max(c->sm_count / 2, 1)));
  tc_xh_kernel<<<grid, kXThreads, smem, stream>>>(P);
  if ((e = cudaGetLastError()) != cudaSuccess) {
    set_error(std::string("kvx_map: cross-head launch: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

}  // namespace kvx
