// Centred second-moment blocks on the tensor cores, for the ridge fit (Sec. 3.1, Eq. Wstar:
// Xc^T Xc and Xc^T Yc) and the single-source R^2 probe (Sec. 2.3).  An operand is one
// (side, layer, K|V, head) of a bf16 cache over the N = B T calibration tokens: keys with
// the RoPE stripped (Sec. 3.3), values as stored, centred by the column means.  A block is
//   G[i][j] = sum_n (a_n[i] - mean_a[i]) (b_n[j] - mean_b[j]),   i, j < 128.
//
// Three kernels:
// 1. gram_pack_kernel<0> (column sums): thread = two tokens x eight RoPE pairs of one
//    64-token chunk; it walks the K|V heads of one slot, strips the keys in fp32 (cos / sin
//    once per token and pair), reduces the 64 tokens across the warp in fp32 and adds the
//    chunk's sums into fp64.
// 2. gram_pack_kernel<1> (pack): the same walk, centring by the fp32 means and splitting
//    each centred value x into bf16 hi + lo (hi = bf16(x), lo = bf16(x - hi); |x - hi - lo|
//    <= 2^-17 |x|), written transposed ([channel][token]) into a workspace
//    [slot][K|V][head][hi|lo][128][tokens] so that an operand tile (128 channels x 64
//    tokens) is one TMA box in the tensor cores' K-major 128-byte-swizzled layout.
// 3. gram_tc_kernel: persistent, one CTA per SM; work unit = one A operand against one or
//    two B operands (N = 128 or 256).  Per 64-token stage the A hi/lo and B hi/lo tiles
//    land by TMA and one thread issues, per 16-token step, the four MMAs of
//    (A_hi + A_lo)(B_hi + B_lo) (tcgen05.mma kind::f16, M = 128, fp32 accumulators in
//    TMEM): the products of bf16 values are exact, so a block is the fp32-accumulated Gram
//    of the operands hi + lo, each within 2^-17 (relative) of the centred value.  All four terms are
//    needed: without A_lo B_lo a block of X^T X becomes (H + L)^T (H + L) - L^T L, which
//    is indefinite along the null space of a rank-deficient X (N < F, ridge-regularised).
//    Four epilogue warps move each finished accumulator (double-buffered in TMEM) to the
//    fp32 output blocks.
// Centring before the products avoids the cancellation of sum x x^T - N mean mean^T; the
// means come from fp32 chunk sums, and an error e in a mean changes a block only by
// N e e^T (the cross terms vanish because centred columns sum to zero).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <numeric>
#include <string>
#include <vector>

#include "kvx_gram.h"
#include "kvx_internal.h"
#include "kvx_ptx.cuh"
#include "kvx_rope.cuh"

namespace kvx {
namespace {

using namespace ptx;

constexpr int kGD = 128;                     // head_dim
constexpr int kGChunk = 64;                  // tokens per pack block and per MMA stage
constexpr int kGPackThreads = 256;           // 8 warps: warp = 8 RoPE pairs, lane = 2 tokens
constexpr uint32_t kGPackTile = 2 * kGD * kGChunk * 2;   // hi and lo: 128 channels x 64 tokens, 32 KB
constexpr int kGTrigWords = 2 * 2 * 8 * 8 * 32;           // cos and sin of each thread's 2 x 8 angles

__device__ __forceinline__ int trig_index(int cs, int q, int m, int g, int lane) {
  return (((cs * 2 + q) * 8 + m) * 8 + g) * 32 + lane;
}

constexpr size_t pack_smem_bytes(int mode) {
  return static_cast<size_t>(kGTrigWords) * 4 + (mode == 1 ? 2 * static_cast<size_t>(kGPackTile) : 0);
}

struct PackParams {
  GramCache c[2];
  const int32_t* pos;
  const int32_t* slots;        // [n_slots][2]: side, layer
  double* sums;                // [2][2][L][H][128]
  const float* means;          // [n_slots][2][H][128] (pack)
  double* sumsq;               // [n_slots][2][H] or NULL
  __nv_bfloat16* ws;           // [n_slots][2][H][2][128][np]
  int32_t* status;
  int64_t n0;                  // first token of the chunk (pack) or 0 (sums)
  int64_t n_end;               // tokens past n_end are zero padding
  int32_t np;                  // tokens per workspace row (multiple of 64)
  int32_t B, T, H, Ls, Lt, hf;
  RopeTables rope;
};

__device__ __forceinline__ float rbf(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

__device__ __forceinline__ void greport(int32_t* status, int code) { atomicCAS(status, 0, code); }

__device__ __forceinline__ size_t gsums_index(const PackParams& P, int side, int kv, int layer, int h) {
  const size_t base = side == 0 ? 0 : static_cast<size_t>(2) * P.Ls * P.H * kGD;
  const int L = side == 0 ? P.Ls : P.Lt;
  return base + ((static_cast<size_t>(kv) * L + layer) * P.H + h) * kGD;
}

// grid: (np / 64 chunks, n_slots), 256 threads, pack_smem_bytes(MODE) dynamic shared memory.
// Warp g owns RoPE pairs 8g .. 8g+7 (channels 8g.. and 64+8g..), lane owns tokens 2 lane and
// 2 lane + 1 of the chunk.
template <int MODE>
__global__ void __launch_bounds__(kGPackThreads, 2) gram_pack_kernel(const __grid_constant__ PackParams P) {
  // [2 cos|sin][2 tokens][8 pairs][8 warps][32 lanes] fp32, then (MODE 1) the transpose tiles
  // [2 bufs][2 parts][128 ch][32 token pairs]; each thread reads back only its own angles
  extern __shared__ __align__(16) uint32_t psm[];
  float* trig = reinterpret_cast<float*>(psm);
  uint32_t* tile = psm + kGTrigWords;
  const int g = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int slot = blockIdx.y;
  const int side = __ldg(&P.slots[2 * slot]), layer = __ldg(&P.slots[2 * slot + 1]);
  const GramCache& c = P.c[side];
  const int64_t nbase = P.n0 + static_cast<int64_t>(blockIdx.x) * kGChunk + 2 * lane;
  bool valid[2];
  int64_t off[2];              // token offset within a (layer, head) row: b s_b + t s_t
  const float* w_hi = side == 0 ? P.rope.ws_hi : P.rope.wt_hi;
  const float* w_lo = side == 0 ? P.rope.ws_lo : P.rope.wt_lo;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int64_t n = nbase + q;
    valid[q] = n < P.n_end;
    off[q] = 0;
    int p = 0;
    if (valid[q]) {
      const int b = static_cast<int>(n / P.T), t = static_cast<int>(n % P.T);
      off[q] = b * c.s[1] + static_cast<int64_t>(t) * c.s[3];
      p = __ldg(&P.pos[n]);
      if (p < 0 || p >= (1 << 24)) {
        greport(P.status, KVX_ERR_DEVICE_BOUNDS);
        p = 0;
      }
    }
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      float sv, cv;
      if (P.hf) {   // HF numerics: cos / sin of the fp32 angle, rounded to bf16
        sincosf(__fmul_rn(static_cast<float>(p), w_hi[8 * g + m]), &sv, &cv);
        sv = rbf(sv);
        cv = rbf(cv);
      } else {
        rope_sincos(p, w_hi[8 * g + m], w_lo[8 * g + m], P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi,
                    &sv, &cv);
      }
      trig[trig_index(0, q, m, g, lane)] = cv;
      trig[trig_index(1, q, m, g, lane)] = sv;
    }
  }
  // the walk over (K|V, head), with the next step's loads issued before this step's math
  const int n_it = 2 * P.H;
  uint4 ra[2], rb[2];
  auto load = [&](int step, uint4 (&xa)[2], uint4 (&xb)[2]) {
    const int kv = step >= P.H ? 1 : 0, h = step - kv * P.H;
    const __nv_bfloat16* base = static_cast<const __nv_bfloat16*>(kv ? c.v : c.k) + layer * c.s[0] + h * c.s[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      xa[q] = make_uint4(0, 0, 0, 0);
      xb[q] = make_uint4(0, 0, 0, 0);
      if (valid[q]) {
        const __nv_bfloat16* row = base + off[q];
        xa[q] = __ldg(reinterpret_cast<const uint4*>(row + 8 * g));
        xb[q] = __ldg(reinterpret_cast<const uint4*>(row + 64 + 8 * g));
      }
    }
  };
  load(0, ra, rb);
  for (int it = 0; it < n_it; ++it) {
    const int kv = it >= P.H ? 1 : 0, h = it - kv * P.H;
    uint4 na[2], nb[2];
    if (it + 1 < n_it) load(it + 1, na, nb);
    {
      // the two tokens' eight pairs, stripped (keys), as fp32
      float va[2][8], vb[2][8];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint32_t wa[4] = {ra[q].x, ra[q].y, ra[q].z, ra[q].w}, wb[4] = {rb[q].x, rb[q].y, rb[q].z, rb[q].w};
#pragma unroll
        for (int m = 0; m < 8; ++m) {
          const float a = (m & 1) ? bf16_hi(wa[m >> 1]) : bf16_lo(wa[m >> 1]);
          const float b = (m & 1) ? bf16_hi(wb[m >> 1]) : bf16_lo(wb[m >> 1]);
          if (kv == 0 && P.hf) {   // the HF strip: each product and sum rounded to bf16
            const float cv = trig[trig_index(0, q, m, g, lane)], sv = trig[trig_index(1, q, m, g, lane)];
            va[q][m] = rbf(__fadd_rn(rbf(__fmul_rn(a, cv)), rbf(__fmul_rn(b, sv))));
            vb[q][m] = rbf(__fsub_rn(rbf(__fmul_rn(b, cv)), rbf(__fmul_rn(a, sv))));
          } else if (kv == 0) {   // rotation by -t omega: a' = a c + b s, b' = b c - a s
            const float cv = trig[trig_index(0, q, m, g, lane)], sv = trig[trig_index(1, q, m, g, lane)];
            va[q][m] = __fmaf_rn(a, cv, __fmul_rn(b, sv));
            vb[q][m] = __fmaf_rn(b, cv, -__fmul_rn(a, sv));
          } else {
            va[q][m] = a;
            vb[q][m] = b;
          }
        }
      }
      if (MODE == 0) {
        // 64-token sums in fp32 across the warp, then one fp64 atomic per channel
        float s[16];
#pragma unroll
        for (int m = 0; m < 8; ++m) {
          s[m] = va[0][m] + va[1][m];
          s[8 + m] = vb[0][m] + vb[1][m];
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1)
#pragma unroll
          for (int m = 0; m < 16; ++m) s[m] += __shfl_xor_sync(0xffffffffu, s[m], d);
        if (lane < 16) {
          float v = s[0];
#pragma unroll
          for (int m = 1; m < 16; ++m)
            if (lane == m) v = s[m];
          const int ch = lane < 8 ? 8 * g + lane : 64 + 8 * g + (lane - 8);
          atomicAdd(&P.sums[gsums_index(P, side, kv, layer, h) + ch], static_cast<double>(v));
        }
      } else {
        const float* means = P.means + ((static_cast<size_t>(slot) * 2 + kv) * P.H + h) * kGD;
        uint32_t* tb = tile + (it & 1) * (kGPackTile / 4);
        float sq = 0.f;
#pragma unroll
        for (int m = 0; m < 8; ++m) {
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            const int ch = half * 64 + 8 * g + m;
            const float mean = __ldg(&means[ch]);
            float x0 = half ? vb[0][m] : va[0][m], x1 = half ? vb[1][m] : va[1][m];
            x0 = valid[0] ? x0 - mean : 0.f;
            x1 = valid[1] ? x1 - mean : 0.f;
            sq = __fmaf_rn(x0, x0, __fmaf_rn(x1, x1, sq));
            const uint32_t hi = pack_bf16x2(x0, x1);
            const uint32_t lo = pack_bf16x2(x0 - bf16_lo(hi), x1 - bf16_hi(hi));
            tb[ch * 32 + lane] = hi;
            tb[(kGD + ch) * 32 + lane] = lo;
          }
        }
        if (P.sumsq != nullptr) {
#pragma unroll
          for (int d = 16; d >= 1; d >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, d);
          if (lane == 0) atomicAdd(&P.sumsq[(static_cast<size_t>(slot) * 2 + kv) * P.H + h], static_cast<double>(sq));
        }
        __syncthreads();
        // 256 rows (hi 0..127, lo 128..255) of 128 bytes: 16-byte pieces, 4 rows per warp
        __nv_bfloat16* dst = P.ws + ((static_cast<size_t>(slot) * 2 + kv) * P.H + h) * (2 * kGD) * static_cast<size_t>(P.np) +
                             static_cast<size_t>(blockIdx.x) * kGChunk;
#pragma unroll
        for (int r = 0; r < 8; ++r) {
          const int piece = r * kGPackThreads + threadIdx.x;
          const int row = piece >> 3, seg = piece & 7;
          const uint4 v = *reinterpret_cast<const uint4*>(tb + row * 32 + seg * 4);
          *reinterpret_cast<uint4*>(dst + static_cast<size_t>(row) * P.np + seg * 8) = v;
        }
      }
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      ra[q] = na[q];
      rb[q] = nb[q];
    }
  }
}

// fp32 column means [slot][K|V][head][128] of the slots, from the fp64 sums.
__global__ void gram_means_kernel(const __grid_constant__ PackParams P, float* means, int n_slots) {
  const int64_t n = static_cast<int64_t>(n_slots) * 2 * P.H * kGD;
  const double inv_n = 1.0 / static_cast<double>(static_cast<int64_t>(P.B) * P.T);
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int ch = static_cast<int>(i % kGD);
    const int64_t r = i / kGD;
    const int h = static_cast<int>(r % P.H), kv = static_cast<int>((r / P.H) % 2), slot = static_cast<int>(r / (2 * P.H));
    const int side = P.slots[2 * slot], layer = P.slots[2 * slot + 1];
    means[i] = static_cast<float>(P.sums[gsums_index(P, side, kv, layer, h) + ch] * inv_n);
  }
}

// ------------------------------------------------------------ tensor-core blocks --

constexpr int kGThreads = 256;               // warp 0 TMA, warp 1 TMEM + MMA, warps 4-7 epilogue
constexpr int kGFirstEpi = 4;
constexpr int kGStages = 2;
constexpr uint32_t kGTileBytes = 128 * 128;  // 128 rows (channels) x 64 tokens bf16
// stage: A hi | A lo | B hi (b0, b1) | B lo (b0, b1)
constexpr uint32_t kGStageBytes = 6 * kGTileBytes;
constexpr uint32_t kGAccCols = 256;
constexpr uint32_t kGTmemCols = 512;
constexpr size_t kGSmemLimit = 232448;

constexpr size_t gram_smem_bytes() {
  return static_cast<size_t>(kGStages) * kGStageBytes + (2 * kGStages + 4 + 1) * 8 + 16;
}
static_assert(gram_smem_bytes() <= kGSmemLimit, "Gram kernel shared memory exceeds the per-CTA limit");

// One unit: rows of the workspace tensor map (hi part; lo = row + 128) of the A operand and
// of one or two B operands (b_row1 < 0: N = 128), and the output blocks.
struct GramUnit {
  int32_t a_row, b_row0, b_row1, pad;
  float* out0;
  float* out1;
};

struct GramTcParams {
  CUtensorMap tm;              // workspace as 2D {np tokens, rows}, box 64 x 128, 128-byte swizzle
  const GramUnit* units;
  int32_t* status;
  int32_t n_units, n_kc;       // units, 64-token stages per unit
  int32_t accumulate;          // add into the output blocks (token chunks after the first)
};

__device__ __forceinline__ void tc_mma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tmem_ld_x32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
        "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
        "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr)
      : "memory");
}

__global__ void __launch_bounds__(kGThreads, 1) gram_tc_kernel(const __grid_constant__ GramTcParams P) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) greport(P.status, KVX_ERR_UNSUPPORTED);
    return;
  }
  uint8_t* stages = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(kGStages) * kGStageBytes);
  uint64_t* empty = full + kGStages;
  uint64_t* accf = empty + kGStages;           // [2] accumulator complete
  uint64_t* acce = accf + 2;                   // [2] accumulator drained (4 epilogue warps)
  uint64_t* drain = acce + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  volatile uint32_t* abort_flag = tmem_holder + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kGStages; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accf[i]), 1);
      mbar_init(smem_u32(&acce[i]), 4);
    }
    mbar_init(smem_u32(&drain[0]), 1);
    *abort_flag = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(kGTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int n_units = P.n_units, n_kc = P.n_kc;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer ----
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();
      uint32_t sn = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        const GramUnit un = P.units[u];
        const bool two = un.b_row1 >= 0;
        for (int kc = 0; kc < n_kc; ++kc, ++sn) {
          const int st = static_cast<int>(sn % kGStages);
          const uint32_t round = sn / kGStages;
          if (round > 0 &&
              !wait_bar(smem_u32(&empty[st]), (round - 1) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT)) {
            ok = false;
            break;
          }
          const uint32_t bar = smem_u32(&full[st]);
          const uint32_t s0 = smem_u32(stages + static_cast<size_t>(st) * kGStageBytes);
          const int x = kc * kGChunk;
          mbar_expect_tx(bar, (two ? 6u : 4u) * kGTileBytes);
          tma_load_2d(s0, &P.tm, bar, x, un.a_row, pol);
          tma_load_2d(s0 + kGTileBytes, &P.tm, bar, x, un.a_row + kGD, pol);
          tma_load_2d(s0 + 2 * kGTileBytes, &P.tm, bar, x, un.b_row0, pol);
          tma_load_2d(s0 + 4 * kGTileBytes, &P.tm, bar, x, un.b_row0 + kGD, pol);
          if (two) {
            tma_load_2d(s0 + 3 * kGTileBytes, &P.tm, bar, x, un.b_row1, pol);
            tma_load_2d(s0 + 5 * kGTileBytes, &P.tm, bar, x, un.b_row1 + kGD, pol);
          }
        }
      }
      if (!ok) {   // the most recent loads may still be landing
        const uint32_t first = sn > static_cast<uint32_t>(kGStages) ? sn - kGStages : 0;
        for (uint32_t i = first; i < sn; ++i) drain_wait(smem_u32(&full[i % kGStages]), (i / kGStages) & 1u);
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer ----
    if (lane == 0) {
      uint32_t si = 0, acc_n = 0;
      bool ok = true, issued = false;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x, ++acc_n) {
        const bool two = P.units[u].b_row1 >= 0;
        const uint32_t idesc = two ? make_idesc(128, 256) : make_idesc(128, 128);
        const uint32_t buf = acc_n & 1u;
        if (acc_n >= 2 &&
            !wait_bar(smem_u32(&acce[buf]), ((acc_n >> 1) - 1) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + buf * kGAccCols;
        for (int kc = 0; kc < n_kc; ++kc, ++si) {
          const uint32_t st = si % kGStages;
          if (!wait_bar(smem_u32(&full[st]), (si / kGStages) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_hi = smem_u32(stages + static_cast<size_t>(st) * kGStageBytes);
          const uint32_t a_lo = a_hi + kGTileBytes;
          const uint32_t b_hi = a_hi + 2 * kGTileBytes;
          const uint32_t b_lo = a_hi + 4 * kGTileBytes;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {   // 16 tokens = 32 bytes along the swizzled row
            tc_mma_ss(d_tmem, sw128_desc(a_hi + kk * 32), sw128_desc(b_hi + kk * 32), idesc, (kc | kk) != 0);
            tc_mma_ss(d_tmem, sw128_desc(a_hi + kk * 32), sw128_desc(b_lo + kk * 32), idesc, 1u);
            tc_mma_ss(d_tmem, sw128_desc(a_lo + kk * 32), sw128_desc(b_hi + kk * 32), idesc, 1u);
            tc_mma_ss(d_tmem, sw128_desc(a_lo + kk * 32), sw128_desc(b_lo + kk * 32), idesc, 1u);
          }
          issued = true;
          tc_commit(smem_u32(&empty[st]));
        }
        if (ok) tc_commit(smem_u32(&accf[buf]));
      }
      if (issued || !ok) {
        tc_commit(smem_u32(&drain[0]));
        drain_wait(smem_u32(&drain[0]), 0);
      }
    }
  } else if (warp >= kGFirstEpi) {
    // ---------------------------------------------------------------- epilogue ----
    const int q = warp & 3;                      // TMEM lane quarter = rows 32q .. 32q+31
    const int r = q * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    uint32_t acc_n = 0;
    for (int u = blockIdx.x; u < n_units; u += gridDim.x, ++acc_n) {
      const GramUnit un = P.units[u];
      const uint32_t buf = acc_n & 1u;
      const bool w_ok = wait_bar(smem_u32(&accf[buf]), (acc_n >> 1) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT);
      if (!__all_sync(0xffffffffu, w_ok)) break;
      tc_fence_after();
      const int nb = un.b_row1 >= 0 ? 2 : 1;
      for (int j = 0; j < nb; ++j) {
        float* out = (j ? un.out1 : un.out0) + static_cast<size_t>(r) * kGD;
#pragma unroll 1
        for (int c0 = 0; c0 < kGD; c0 += 32) {
          uint32_t v[32];
          tmem_ld_x32(tmem_base + lane_addr + buf * kGAccCols + j * kGD + c0, v);
          float4* o = reinterpret_cast<float4*>(out + c0);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            float4 w = make_float4(__uint_as_float(v[4 * e]), __uint_as_float(v[4 * e + 1]),
                                   __uint_as_float(v[4 * e + 2]), __uint_as_float(v[4 * e + 3]));
            if (P.accumulate) {
              const float4 old = o[e];
              w.x += old.x;
              w.y += old.y;
              w.z += old.z;
              w.w += old.w;
            }
            o[e] = w;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&acce[buf]));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kGTmemCols)
                 : "memory");
  }
}

kvx_status cuda_fail(const char* what, cudaError_t e) {
  set_error(std::string(what) + ": " + cudaGetErrorString(e));
  return e == cudaErrorMemoryAllocation ? KVX_ERR_OOM : KVX_ERR_CUDA;
}

PackParams pack_params(const GramSpec& s) {
  PackParams P;
  std::memset(&P, 0, sizeof(P));
  P.c[0] = s.cache[0];
  P.c[1] = s.cache[1];
  P.pos = s.pos;
  P.sums = s.sums;
  P.sumsq = s.sumsq;
  P.status = s.status;
  P.B = s.B;
  P.T = s.T;
  P.H = s.H;
  P.Ls = s.Ls;
  P.Lt = s.Lt;
  P.hf = s.hf;
  P.rope = s.rope;
  return P;
}

std::vector<int32_t> slot_table(const GramSpec& s) {
  std::vector<int32_t> t(2 * s.slot_side.size());
  for (size_t i = 0; i < s.slot_side.size(); ++i) {
    t[2 * i] = s.slot_side[i];
    t[2 * i + 1] = s.slot_layer[i];
  }
  return t;
}

}  // namespace

PhaseTimer::~PhaseTimer() {
  for (cudaEvent_t e : ev_) cudaEventDestroy(e);
}

void PhaseTimer::begin(int phase) {
  cudaEvent_t a = nullptr, b = nullptr;
  if (cudaEventCreate(&a) != cudaSuccess) return;
  if (cudaEventCreate(&b) != cudaSuccess) {
    cudaEventDestroy(a);
    return;
  }
  cudaEventRecord(a, stream_);
  ev_.push_back(a);
  ev_.push_back(b);
  phase_.push_back(phase);
  open_ = static_cast<int>(phase_.size()) - 1;
}

void PhaseTimer::end() {
  if (open_ < 0) return;
  cudaEventRecord(ev_[2 * open_ + 1], stream_);
  open_ = -1;
}

namespace {
thread_local float g_phase_ms[4] = {0.f, 0.f, 0.f, 0.f};
}

void PhaseTimer::finish() {
  float ms[4] = {0.f, 0.f, 0.f, 0.f};
  for (size_t i = 0; i < phase_.size(); ++i) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, ev_[2 * i], ev_[2 * i + 1]) == cudaSuccess && phase_[i] >= 0 && phase_[i] < 4)
      ms[phase_[i]] += t;
  }
  for (int i = 0; i < 4; ++i) g_phase_ms[i] = ms[i];
}

size_t gram_fixed_bytes(const GramSpec& spec, size_t n_blocks) {
  const size_t n_slots = spec.slot_side.size();
  auto al = [](size_t n) { return (n + 255) / 256 * 256; };
  return al(n_slots * 2 * 4) /* gram_sums slot table */ + al(n_blocks * sizeof(GramUnit)) + al(n_slots * 2 * 4) +
         al(n_slots * 2 * static_cast<size_t>(spec.H) * kGD * 4);
}

size_t gram_bytes_per_token(const GramSpec& spec) {
  return spec.slot_side.size() * 2 * static_cast<size_t>(spec.H) * 2 * kGD * 2;
}

kvx_status gram_sums(const GramSpec& spec, cudaStream_t stream, PhaseTimer* timer, Scratch* scratch) {
  const int n_slots = static_cast<int>(spec.slot_side.size());
  if (n_slots == 0) return KVX_OK;
  const int64_t N = static_cast<int64_t>(spec.B) * spec.T;
  const std::vector<int32_t> tab = slot_table(spec);
  int32_t* d_tab = nullptr;
  cudaError_t e;
  const bool own = !(scratch && scratch->p);
  if (own) {
    if ((e = cudaMallocAsync(reinterpret_cast<void**>(&d_tab), tab.size() * 4, stream)) != cudaSuccess)
      return cuda_fail("column sums: workspace", e);
  } else if (!(d_tab = reinterpret_cast<int32_t*>(scratch->take(tab.size() * 4)))) {
    set_error("column sums: workspace too small");
    return KVX_ERR_INVALID_ARG;
  }
  kvx_status r = KVX_OK;
  if ((e = cudaMemcpyAsync(d_tab, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice, stream)) != cudaSuccess) {
    r = cuda_fail("column sums: slot table", e);
  } else {
    PackParams P = pack_params(spec);
    P.slots = d_tab;
    P.n0 = 0;
    P.n_end = N;
    P.np = 0;
    const dim3 grid(static_cast<unsigned>((N + kGChunk - 1) / kGChunk), static_cast<unsigned>(n_slots));
    if (timer) timer->begin(0);
    gram_pack_kernel<0><<<grid, kGPackThreads, pack_smem_bytes(0), stream>>>(P);
    if (timer) timer->end();
    if ((e = cudaGetLastError()) != cudaSuccess) r = cuda_fail("column sums: launch", e);
  }
  if (own) cudaFreeAsync(d_tab, stream);
  return r;
}

kvx_status gram_blocks(const GramSpec& spec, const std::vector<GramBlock>& blocks, size_t ws_budget,
                       cudaStream_t stream, PhaseTimer* timer, Scratch* scratch) {
  if (blocks.empty()) return KVX_OK;
  auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
  if (!encode) {
    set_error("Gram blocks: cuTensorMapEncodeTiled unavailable");
    return KVX_ERR_CUDA;
  }
  const int n_slots = static_cast<int>(spec.slot_side.size());
  const int64_t rows = static_cast<int64_t>(n_slots) * 2 * spec.H * 2 * kGD;
  if (rows > INT_MAX - 2 * kGD) {
    set_error("Gram blocks: too many operands");
    return KVX_ERR_UNSUPPORTED;
  }
  const int64_t N = static_cast<int64_t>(spec.B) * spec.T;
  const int64_t np_full = (N + kGChunk - 1) / kGChunk * kGChunk;
  const bool own = !(scratch && scratch->p);
  if (!own) {   // the fixed pieces come first; the packed operands get the rest
    const size_t fixed = gram_fixed_bytes(spec, blocks.size()) - (n_slots * 2 * 4 + 255) / 256 * 256;
    ws_budget = scratch->bytes > fixed + 256 ? scratch->bytes - fixed - 256 : 0;
  }
  const int64_t np_fit = static_cast<int64_t>(ws_budget / (static_cast<size_t>(rows) * 2)) / kGChunk * kGChunk;
  if (np_fit < kGChunk) {
    set_error(own ? "Gram blocks: the workspace budget holds less than 64 tokens of the operands"
                  : "Gram blocks: the caller's workspace holds less than 64 tokens of the operands");
    return own ? KVX_ERR_OOM : KVX_ERR_INVALID_ARG;
  }
  const int64_t np = std::min<int64_t>(std::min(np_full, np_fit), INT_MAX / 2 / kGChunk * kGChunk);
  const int64_t n_chunks = (N + np - 1) / np;

  // units: blocks sorted by (K|V, head, A operand, B operand); consecutive blocks that share
  // the A operand run as one N = 256 unit
  std::vector<size_t> order(blocks.size());
  std::iota(order.begin(), order.end(), 0);
  std::sort(order.begin(), order.end(), [&](size_t x, size_t y) {
    const GramBlock &p = blocks[x], &q = blocks[y];
    if (p.kv != q.kv) return p.kv < q.kv;
    if (p.h != q.h) return p.h < q.h;
    if (p.a_slot != q.a_slot) return p.a_slot < q.a_slot;
    if (p.b_slot != q.b_slot) return p.b_slot < q.b_slot;
    return p.hb < q.hb;
  });
  auto row_of = [&](int slot, int kv, int h) {
    return static_cast<int32_t>(((static_cast<int64_t>(slot) * 2 + kv) * spec.H + h) * 2 * kGD);
  };
  std::vector<GramUnit> units;
  for (size_t i = 0; i < order.size();) {
    const GramBlock& p = blocks[order[i]];
    GramUnit u{};
    u.a_row = row_of(p.a_slot, p.kv, p.h);
    u.b_row0 = row_of(p.b_slot, p.kv, p.hb < 0 ? p.h : p.hb);
    u.b_row1 = -1;
    u.out0 = p.out;
    u.out1 = nullptr;
    if (i + 1 < order.size()) {
      const GramBlock& q = blocks[order[i + 1]];
      if (q.kv == p.kv && q.h == p.h && q.a_slot == p.a_slot) {
        u.b_row1 = row_of(q.b_slot, q.kv, q.hb < 0 ? q.h : q.hb);
        u.out1 = q.out;
        ++i;
      }
    }
    ++i;
    units.push_back(u);
  }
  if (units.size() > static_cast<size_t>(INT_MAX)) {
    set_error("Gram blocks: too many blocks");
    return KVX_ERR_UNSUPPORTED;
  }
  const std::vector<int32_t> tab = slot_table(spec);
  auto al = [](size_t n) { return (n + 255) / 256 * 256; };
  const size_t ws_bytes = static_cast<size_t>(rows) * static_cast<size_t>(np) * 2;
  const size_t units_off = al(ws_bytes);
  const size_t tab_off = units_off + al(units.size() * sizeof(GramUnit));
  const size_t means_off = tab_off + al(tab.size() * 4);
  const size_t means_n = static_cast<size_t>(n_slots) * 2 * spec.H * kGD;
  const size_t total = means_off + al(means_n * 4);
  char* mem = nullptr;
  cudaError_t e;
  if (own) {
    if ((e = cudaMallocAsync(reinterpret_cast<void**>(&mem), total, stream)) != cudaSuccess)
      return cuda_fail("Gram blocks: workspace", e);
  } else if (!(mem = scratch->take(total))) {
    set_error("Gram blocks: the caller's workspace is too small");
    return KVX_ERR_INVALID_ARG;
  }
  kvx_status r = KVX_OK;
  do {
    if ((e = cudaMemcpyAsync(mem + units_off, units.data(), units.size() * sizeof(GramUnit), cudaMemcpyHostToDevice,
                             stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(mem + tab_off, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice, stream)) !=
            cudaSuccess) {
      r = cuda_fail("Gram blocks: tables", e);
      break;
    }
    GramTcParams G;
    std::memset(&G, 0, sizeof(G));
    {
      const cuuint64_t dims[2] = {static_cast<cuuint64_t>(np), static_cast<cuuint64_t>(rows)};
      const cuuint64_t str[1] = {static_cast<cuuint64_t>(np) * 2};
      const cuuint32_t box[2] = {kGChunk, 128};
      const cuuint32_t ones[2] = {1, 1};
      CUresult cr = encode(&G.tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, mem, dims, str, box, ones,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (cr != CUDA_SUCCESS) {
        set_error("Gram blocks: workspace tensor map rejected");
        r = KVX_ERR_CUDA;
        break;
      }
    }
    G.units = reinterpret_cast<const GramUnit*>(mem + units_off);
    G.status = spec.status;
    G.n_units = static_cast<int32_t>(units.size());
    const size_t gsmem = gram_smem_bytes();
    if ((e = cudaFuncSetAttribute(gram_pack_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(pack_smem_bytes(1)))) != cudaSuccess ||
        (e = cudaFuncSetAttribute(gram_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(gsmem))) != cudaSuccess) {
      r = cuda_fail("Gram blocks: shared memory attribute", e);
      break;
    }
    PackParams P = pack_params(spec);
    P.slots = reinterpret_cast<const int32_t*>(mem + tab_off);
    P.ws = reinterpret_cast<__nv_bfloat16*>(mem);
    P.np = static_cast<int32_t>(np);
    float* means = reinterpret_cast<float*>(mem + means_off);
    P.means = means;
    gram_means_kernel<<<static_cast<unsigned>(std::min<size_t>((means_n + 255) / 256, 4096)), 256, 0, stream>>>(
        P, means, n_slots);
    const int grid = static_cast<int>(std::min<int64_t>(static_cast<int64_t>(units.size()), std::max(spec.sm_count, 1)));
    for (int64_t ch = 0; ch < n_chunks && r == KVX_OK; ++ch) {
      P.n0 = ch * np;
      P.n_end = std::min(N, P.n0 + np);
      const int64_t kc = (P.n_end - P.n0 + kGChunk - 1) / kGChunk;
      if (timer) timer->begin(1);
      gram_pack_kernel<1><<<dim3(static_cast<unsigned>(kc), static_cast<unsigned>(n_slots)), kGPackThreads,
                            pack_smem_bytes(1), stream>>>(P);
      if (timer) timer->end();
      G.n_kc = static_cast<int32_t>(kc);
      G.accumulate = ch > 0 ? 1 : 0;
      if (timer) timer->begin(2);
      gram_tc_kernel<<<grid, kGThreads, gsmem, stream>>>(G);
      if (timer) timer->end();
      if ((e = cudaGetLastError()) != cudaSuccess) r = cuda_fail("Gram blocks: launch", e);
    }
  } while (false);
  if (own) cudaFreeAsync(mem, stream);
  return r;
}

}  // namespace kvx

extern "C" KVX_API kvx_status kvx_last_phase_ms(float* ms) {
  if (!ms) return KVX_ERR_INVALID_ARG;
  for (int i = 0; i < 4; ++i) ms[i] = kvx::g_phase_ms[i];
  return KVX_OK;
}
