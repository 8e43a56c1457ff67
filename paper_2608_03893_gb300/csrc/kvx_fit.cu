// Ridge fit of the per-head mapper on the GPU (Sec. 3.1, Eq. Wstar; keys RoPE-stripped
// on both sides, Sec. 3.3).  For every target layer l, K|V and head h, over the N =
// B * T calibration tokens:
//   X = [x_{sel[l][0]} || ... || x_{sel[l][k-1]}]   (F = k d features; source keys with
//       the source RoPE stripped, source values as they are),
//   Y = head h of target layer l (target keys with the target RoPE stripped, values),
//   Xc, Yc centred by their column means,
//   W = (Xc^T Xc + lambda I)^{-1} Xc^T Yc,   b = mean(Y) - mean(X) W.
// bf16 caches, head_dim 128, half-split pairs.
//
// Three kernels, all in this file:
// 1. fit_mean_kernel: fp64 column sums of every (side, K|V, layer, head) over the tokens;
//    a thread owns one RoPE pair (channels i and i + 64) of one row and a chunk of tokens,
//    strips the rotation in fp32 and adds into fp64 with one atomic per chunk.
// 2. fit_gram_kernel: one CTA per 128 x 128 block: a (source layer, source layer) block of
//    Xc^T Xc, computed once for every target layer whose selection holds both layers, or
//    a (source layer, target layer) block of Xc^T Yc; the token loop stages 32-token tiles of both
//    operands in shared memory already stripped and centred (fp32), and 256 threads each
//    accumulate an 8 x 8 register tile with FFMA.  fp32 accumulation of centred values.
// 3. fit_solve_kernel: one CTA per system at a time (persistent); the block grid is
//    widened to fp64 into a per-CTA scratch matrix, lambda added, factorised by a blocked
//    right-looking Cholesky (32-column panels: diagonal block in shared memory, panel by
//    forward substitution, trailing update), then the two triangular solves for the d
//    right-hand sides and the bias; W and b are written in fp32.
// kvx_fit_ridge runs them on the caller's stream, with stream-ordered workspace, and
// synchronises before it returns (the fit is an offline step).
#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <string>
#include <vector>

#include "kvx_internal.h"
#include "kvx_ptx.cuh"
#include "kvx_rope.cuh"

namespace kvx {
namespace {

using namespace ptx;

constexpr int kFD = 128;            // head_dim
constexpr int kFPairs = kFD / 2;    // RoPE pairs per head
constexpr int kFChunk = 1024;       // tokens per block of the mean kernel
constexpr int kGTok = 32;           // tokens per stage of the Gram kernel
constexpr int kNB = 32;             // Cholesky panel width

// Where one operand row lives: side 0 = source (selected layers), 1 = target.
struct FitCache {
  const __nv_bfloat16* k;
  const __nv_bfloat16* v;
  int64_t s[4];                     // strides (layer, batch, head, token), elements
};

struct FitParams {
  FitCache src, tgt;
  const int32_t* pos;               // [B][T]
  const int32_t* sel;               // [L_t][k]
  int32_t Ls, Lt, H, k, B, T;
  RopeTables rope;
  double* sums;                     // [2 sides][2 kv][L][H][128]: side 0 L = L_s, side 1 L = L_t
  float* gram;                      // [2][H][n_pairs][128][128]: source-pair blocks
  const int32_t* pairs;             // [n_pairs][2] source layers (sa >= sb)
  const int32_t* pair_of;           // [L_t][k][k] pair of block (bi, bj), bi >= bj
  int32_t n_pairs;
  float* xty;                       // [L_t][2][H][k][128][128]
  double* scratch;                  // per CTA: F x F matrix + F x 128 right-hand sides
  float* W;                         // [L_t][2][H][F][128]
  float* b;                         // [L_t][2][H][128]
  double lambda;
  int32_t* status;
};

__device__ __forceinline__ size_t sums_index(const FitParams& P, int side, int kv, int layer, int h) {
  const size_t base = side == 0 ? 0 : static_cast<size_t>(2) * P.Ls * P.H * kFD;
  const int L = side == 0 ? P.Ls : P.Lt;
  return base + ((static_cast<size_t>(kv) * L + layer) * P.H + h) * kFD;
}

// Token n (0 .. B*T-1) of row (layer, head) of one cache, RoPE pair i: the pair's two
// channels as stored, and the position of the token.
__device__ __forceinline__ const __nv_bfloat16* row_ptr(const FitCache& c, int kv, int layer, int h, int b, int t) {
  return (kv ? c.v : c.k) + layer * c.s[0] + b * c.s[1] + h * c.s[2] + static_cast<int64_t>(t) * c.s[3];
}

__device__ __forceinline__ void report_fit(int32_t* status, int code) { atomicCAS(status, 0, code); }

// Keys: the stored pair (a, b) rotated by -t omega_i (strip); values unchanged.
__device__ __forceinline__ void strip_pair(float a, float b, float c, float s, float* ra, float* rb) {
  *ra = __fmaf_rn(a, c, __fmul_rn(b, s));
  *rb = __fmaf_rn(b, c, -__fmul_rn(a, s));
}

// --------------------------------------------------------------- column sums --
// grid: (token chunks, rows), row = ((side * 2 + kv) * Lmax + layer) * H + h; 64 threads.
__global__ void __launch_bounds__(kFPairs) fit_mean_kernel(const __grid_constant__ FitParams P, int Lmax) {
  const int row = blockIdx.y;
  const int h = row % P.H;
  const int rest = row / P.H;
  const int layer = rest % Lmax;
  const int sk = rest / Lmax;            // side * 2 + kv
  const int side = sk >> 1, kv = sk & 1;
  if (layer >= (side == 0 ? P.Ls : P.Lt)) return;
  const FitCache& c = side == 0 ? P.src : P.tgt;
  const int i = threadIdx.x;             // pair: channels i and i + 64
  const float* w_hi = side == 0 ? P.rope.ws_hi : P.rope.wt_hi;
  const float* w_lo = side == 0 ? P.rope.ws_lo : P.rope.wt_lo;
  const int64_t N = static_cast<int64_t>(P.B) * P.T;
  const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kFChunk;
  const int64_t n1 = min(N, n0 + kFChunk);
  double sa = 0.0, sb = 0.0;
  for (int64_t n = n0; n < n1; ++n) {
    const int b = static_cast<int>(n / P.T), t = static_cast<int>(n % P.T);
    const __nv_bfloat16* r = row_ptr(c, kv, layer, h, b, t);
    float a = __bfloat162float(r[i]), bb = __bfloat162float(r[i + kFPairs]);
    if (kv == 0) {
      int p = __ldg(&P.pos[n]);
      if (p < 0 || p >= (1 << 24)) {
        report_fit(P.status, KVX_ERR_DEVICE_BOUNDS);
        p = 0;
      }
      float s, cs;
      rope_sincos(p, w_hi[i], w_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi, &s, &cs);
      strip_pair(a, bb, cs, s, &a, &bb);
    }
    sa += a;
    sb += bb;
  }
  double* out = P.sums + sums_index(P, side, kv, layer, h);
  atomicAdd(&out[i], sa);
  atomicAdd(&out[i + kFPairs], sb);
}

// ------------------------------------------------------------- Gram blocks --
// grid: (n_pairs + L_t k, 2 H), 256 threads, 33 KB shared memory.  x < n_pairs: the
// source-pair block (pairs[x][0], pairs[x][1]) of Xc^T Xc; otherwise the block (l, bi) of
// Xc^T Yc, x - n_pairs = l k + bi.
struct Operand {
  const FitCache* c;
  int side, layer;
};

// Stage tokens n0 .. n0+31 of one operand (head h, K|V kv) into dst[32][128] as fp32,
// keys stripped, centred by `mean` (fp32 [128]); rows past N are zero.
__device__ __forceinline__ void stage_tile(const FitParams& P, const Operand& o, int kv, int h, int64_t n0,
                                           const float* mean, float* dst) {
  const int i = threadIdx.x & (kFPairs - 1);      // pair
  const int t0 = threadIdx.x >> 6;                // 0..3
  const int64_t N = static_cast<int64_t>(P.B) * P.T;
  const float* w_hi = o.side == 0 ? P.rope.ws_hi : P.rope.wt_hi;
  const float* w_lo = o.side == 0 ? P.rope.ws_lo : P.rope.wt_lo;
#pragma unroll 2
  for (int m = 0; m < kGTok / 4; ++m) {
    const int tt = t0 + 4 * m;
    const int64_t n = n0 + tt;
    float a = 0.f, bb = 0.f;
    if (n < N) {
      const int b = static_cast<int>(n / P.T), t = static_cast<int>(n % P.T);
      const __nv_bfloat16* r = row_ptr(*o.c, kv, o.layer, h, b, t);
      a = __bfloat162float(r[i]);
      bb = __bfloat162float(r[i + kFPairs]);
      if (kv == 0) {
        int p = __ldg(&P.pos[n]);
        if (p < 0 || p >= (1 << 24)) p = 0;       // reported by the mean kernel
        float s, cs;
        rope_sincos(p, w_hi[i], w_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi, &s, &cs);
        strip_pair(a, bb, cs, s, &a, &bb);
      }
      a -= mean[i];
      bb -= mean[i + kFPairs];
    }
    dst[tt * kFD + i] = a;
    dst[tt * kFD + i + kFPairs] = bb;
  }
}

__global__ void __launch_bounds__(256) fit_gram_kernel(const __grid_constant__ FitParams P) {
  __shared__ __align__(16) float ta[kGTok * kFD];
  __shared__ __align__(16) float tb[kGTok * kFD];
  __shared__ float mean_a[kFD], mean_b[kFD];
  const int kv = blockIdx.y / P.H, h = blockIdx.y % P.H;
  const int q = blockIdx.x;
  const bool is_pair = q < P.n_pairs;
  const int l = is_pair ? 0 : (q - P.n_pairs) / P.k, bi = is_pair ? 0 : (q - P.n_pairs) % P.k;
  const Operand oa{&P.src, 0, is_pair ? __ldg(&P.pairs[2 * q]) : __ldg(&P.sel[l * P.k + bi])};
  const Operand ob = is_pair ? Operand{&P.src, 0, __ldg(&P.pairs[2 * q + 1])} : Operand{&P.tgt, 1, l};
  const int64_t N = static_cast<int64_t>(P.B) * P.T;
  const double inv_n = 1.0 / static_cast<double>(N);
  if (threadIdx.x < kFD) {
    mean_a[threadIdx.x] = static_cast<float>(P.sums[sums_index(P, 0, kv, oa.layer, h) + threadIdx.x] * inv_n);
    mean_b[threadIdx.x] = static_cast<float>(P.sums[sums_index(P, ob.side, kv, ob.layer, h) + threadIdx.x] * inv_n);
  }
  __syncthreads();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;   // output rows 8ty.., columns 8tx..
  float acc[8][8];
#pragma unroll
  for (int x = 0; x < 8; ++x)
#pragma unroll
    for (int y = 0; y < 8; ++y) acc[x][y] = 0.f;
  for (int64_t n0 = 0; n0 < N; n0 += kGTok) {
    stage_tile(P, oa, kv, h, n0, mean_a, ta);
    stage_tile(P, ob, kv, h, n0, mean_b, tb);
    __syncthreads();
#pragma unroll 4
    for (int t = 0; t < kGTok; ++t) {
      const float4 a0 = *reinterpret_cast<const float4*>(&ta[t * kFD + 8 * ty]);
      const float4 a1 = *reinterpret_cast<const float4*>(&ta[t * kFD + 8 * ty + 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&tb[t * kFD + 8 * tx]);
      const float4 b1 = *reinterpret_cast<const float4*>(&tb[t * kFD + 8 * tx + 4]);
      const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int x = 0; x < 8; ++x)
#pragma unroll
        for (int y = 0; y < 8; ++y) acc[x][y] = __fmaf_rn(av[x], bv[y], acc[x][y]);
    }
    __syncthreads();
  }
  float* out = is_pair ? P.gram + ((static_cast<size_t>(kv) * P.H + h) * P.n_pairs + q) * kFD * kFD
                       : P.xty + (((static_cast<size_t>(l) * 2 + kv) * P.H + h) * P.k + bi) * kFD * kFD;
#pragma unroll
  for (int x = 0; x < 8; ++x) {
    float4* o = reinterpret_cast<float4*>(out + static_cast<size_t>(8 * ty + x) * kFD + 8 * tx);
    o[0] = make_float4(acc[x][0], acc[x][1], acc[x][2], acc[x][3]);
    o[1] = make_float4(acc[x][4], acc[x][5], acc[x][6], acc[x][7]);
  }
}

// ------------------------------------------------------------------- solve --
// Persistent: CTA c handles systems c, c + gridDim.x, ...  F = 128 k (k <= 4).  Dynamic
// shared memory: the 32 x 32 diagonal block and the panel below it ((F - 32) x 32), fp64.
constexpr int kNotSpd = 100;        // internal status: a pivot <= 0 (matrix not positive definite)

__global__ void __launch_bounds__(256) fit_solve_kernel(const __grid_constant__ FitParams P) {
  extern __shared__ __align__(16) double fsm[];
  double* D = fsm;                                // [32][32]
  double* Pn = fsm + kNB * kNB;                   // [F - 32][32]
  const int F = P.k * kFD;
  const int tid = threadIdx.x;
  double* A = P.scratch + static_cast<size_t>(blockIdx.x) * (static_cast<size_t>(F) * F + static_cast<size_t>(F) * kFD);
  double* Z = A + static_cast<size_t>(F) * F;     // [F][128]
  const int n_sys = P.Lt * 2 * P.H;
  const double inv_n = 1.0 / (static_cast<double>(P.B) * P.T);
  for (int sys = blockIdx.x; sys < n_sys; sys += gridDim.x) {
    const int h = sys % P.H;
    const int kv = (sys / P.H) & 1;
    const int l = sys / (2 * P.H);
    // 1. A = Xc^T Xc + lambda I (lower triangle) and Z = Xc^T Yc, widened to fp64
    for (int64_t e = tid; e < static_cast<int64_t>(F) * F; e += blockDim.x) {
      const int r = static_cast<int>(e / F), c = static_cast<int>(e % F);
      if (c > r) continue;
      const int bi = r / kFD, bj = c / kFD;
      const int pr = __ldg(&P.pair_of[(l * P.k + bi) * P.k + bj]);   // < 0: stored transposed
      const size_t blk = ((static_cast<size_t>(kv) * P.H + h) * P.n_pairs + (pr >= 0 ? pr : -1 - pr)) * kFD * kFD;
      const float g = pr >= 0 ? P.gram[blk + static_cast<size_t>(r % kFD) * kFD + (c % kFD)]
                              : P.gram[blk + static_cast<size_t>(c % kFD) * kFD + (r % kFD)];
      A[e] = static_cast<double>(g) + (r == c ? P.lambda : 0.0);
    }
    for (int64_t e = tid; e < static_cast<int64_t>(F) * kFD; e += blockDim.x) {
      const int r = static_cast<int>(e / kFD), j = static_cast<int>(e % kFD);
      Z[e] = static_cast<double>(P.xty[(static_cast<size_t>(sys) * P.k + r / kFD) * kFD * kFD +
                                       static_cast<size_t>(r % kFD) * kFD + j]);
    }
    __syncthreads();
    // 2. Cholesky A = L L^T, lower triangle in place, 32-column panels
    for (int c0 = 0; c0 < F; c0 += kNB) {
      for (int e = tid; e < kNB * kNB; e += blockDim.x) D[e] = A[static_cast<size_t>(c0 + e / kNB) * F + c0 + e % kNB];
      __syncthreads();
      if (tid < 32) {                             // one warp factors the diagonal block, lane = row
        for (int j = 0; j < kNB; ++j) {
          if (tid == j) {
            const double d = D[j * kNB + j];
            if (!(d > 0.0)) report_fit(P.status, kNotSpd);
            D[j * kNB + j] = d > 0.0 ? sqrt(d) : 1.0;
          }
          __syncwarp();
          if (tid > j) D[tid * kNB + j] /= D[j * kNB + j];
          __syncwarp();
          if (tid > j)
            for (int m = j + 1; m <= tid; ++m) D[tid * kNB + m] -= D[tid * kNB + j] * D[m * kNB + j];
          __syncwarp();
        }
      }
      __syncthreads();
      for (int e = tid; e < kNB * kNB; e += blockDim.x)
        if (e % kNB <= e / kNB) A[static_cast<size_t>(c0 + e / kNB) * F + c0 + e % kNB] = D[e];
      // panel: rows below the diagonal block, P[r] L_kk^T = A[r][c0 .. c0+31]
      const int rows = F - c0 - kNB;
      for (int rr = tid; rr < rows; rr += blockDim.x) {
        double* arow = A + static_cast<size_t>(c0 + kNB + rr) * F + c0;
        double x[kNB];
#pragma unroll
        for (int c = 0; c < kNB; ++c) {
          double v = arow[c];
#pragma unroll
          for (int m = 0; m < c; ++m) v -= x[m] * D[c * kNB + m];
          x[c] = v / D[c * kNB + c];
        }
#pragma unroll
        for (int c = 0; c < kNB; ++c) {
          arow[c] = x[c];
          Pn[rr * kNB + c] = x[c];
        }
      }
      __syncthreads();
      // trailing update: A[i][j] -= P[i] . P[j] for c0+32 <= j <= i, in 32 x 32 tiles
      const int nt = rows / kNB;
      for (int tile = 0; tile < nt * (nt + 1) / 2; ++tile) {
        int ti = 0;
        while ((ti + 1) * (ti + 2) / 2 <= tile) ++ti;
        const int tj = tile - ti * (ti + 1) / 2;
        const int ii = ti * kNB + (tid >> 3), jj = tj * kNB + (tid & 7) * 4;
        double s[4] = {0.0, 0.0, 0.0, 0.0};
#pragma unroll 8
        for (int m = 0; m < kNB; ++m) {
          const double pi = Pn[ii * kNB + m];
#pragma unroll
          for (int q = 0; q < 4; ++q) s[q] += pi * Pn[(jj + q) * kNB + m];
        }
        double* arow = A + static_cast<size_t>(c0 + kNB + ii) * F + c0 + kNB;
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (jj + q <= ii) arow[jj + q] -= s[q];
      }
      __syncthreads();
    }
    // 3. forward solve L Y = Z, then backward L^T W = Y, in place on Z; thread = right-hand
    //    side column (128 columns, two threads per column split the inner sums)
    const int j = tid & (kFD - 1), half = tid >> 7;
    for (int r = 0; r < F; ++r) {
      const double* lrow = A + static_cast<size_t>(r) * F;
      double sacc = 0.0;
      for (int m = half; m < r; m += 2) sacc += lrow[m] * Z[static_cast<size_t>(m) * kFD + j];
      Pn[tid] = sacc;                                  // scratch: partial sums of both halves
      __syncthreads();
      if (half == 0) Z[static_cast<size_t>(r) * kFD + j] = (Z[static_cast<size_t>(r) * kFD + j] - Pn[j] - Pn[j + kFD]) / lrow[r];
      __syncthreads();
    }
    for (int r = F - 1; r >= 0; --r) {
      double sacc = 0.0;
      for (int m = r + 1 + half; m < F; m += 2) sacc += A[static_cast<size_t>(m) * F + r] * Z[static_cast<size_t>(m) * kFD + j];
      Pn[tid] = sacc;
      __syncthreads();
      if (half == 0)
        Z[static_cast<size_t>(r) * kFD + j] = (Z[static_cast<size_t>(r) * kFD + j] - Pn[j] - Pn[j + kFD]) / A[static_cast<size_t>(r) * F + r];
      __syncthreads();
    }
    // 4. W (fp32) and b = mean(Y) - mean(X) W
    float* Wout = P.W + static_cast<size_t>(sys) * F * kFD;
    for (int64_t e = tid; e < static_cast<int64_t>(F) * kFD; e += blockDim.x) Wout[e] = static_cast<float>(Z[e]);
    if (tid < kFD) {
      double acc = P.sums[sums_index(P, 1, kv, l, h) + tid] * inv_n;
      for (int r = 0; r < F; ++r) {
        const int layer = __ldg(&P.sel[l * P.k + r / kFD]);
        acc -= P.sums[sums_index(P, 0, kv, layer, h) + r % kFD] * inv_n * Z[static_cast<size_t>(r) * kFD + tid];
      }
      P.b[static_cast<size_t>(sys) * kFD + tid] = static_cast<float>(acc);
    }
    __syncthreads();
  }
}

}  // namespace
}  // namespace kvx

extern "C" {

KVX_API kvx_status kvx_fit_ridge(const kvx_fit_config* cfg, const kvx_src* src, const kvx_src* tgt, int32_t batch,
                                 int32_t tokens_per_seq, const int32_t* positions, float* W, float* b,
                                 void* stream) {
  using namespace kvx;
  set_error("");
  auto bad = [](const char* m) {
    set_error(std::string("kvx_fit_ridge: ") + m);
    return KVX_ERR_INVALID_ARG;
  };
  if (!cfg || !src || !tgt || !positions || !W || !b) return bad("NULL argument");
  if (cfg->head_dim != kFD) return bad("head_dim must be 128");
  if (cfg->k < 1 || cfg->k > 4) return bad("k must be in [1, 4]");
  if (cfg->src_layers < 1 || cfg->tgt_layers < 1 || cfg->n_kv_heads < 1 || cfg->k > cfg->src_layers)
    return bad("layer / head counts out of range");
  if (!(cfg->lambda >= 0.0) || !(cfg->src_rope_theta > 1.0) || !(cfg->tgt_rope_theta > 1.0))
    return bad("lambda must be >= 0 and the RoPE bases > 1");
  if (!cfg->selection) return bad("NULL selection");
  for (int64_t i = 0; i < static_cast<int64_t>(cfg->tgt_layers) * cfg->k; ++i)
    if (cfg->selection[i] < 0 || cfg->selection[i] >= cfg->src_layers) return bad("selection entry out of range");
  if (batch < 1 || tokens_per_seq < 1) return bad("batch and tokens_per_seq must be >= 1");
  const kvx_src* cs[2] = {src, tgt};
  for (const kvx_src* c : cs) {
    if (!c->k || !c->v) return bad("NULL cache pointer");
    if ((reinterpret_cast<uintptr_t>(c->k) | reinterpret_cast<uintptr_t>(c->v)) & 15u)
      return bad("cache pointers must be 16-byte aligned");
    for (int i = 0; i < 4; ++i)
      if (c->stride[i] < 0 || c->stride[i] % 8 != 0) return bad("strides must be non-negative multiples of 8");
    if (c->stride[3] < kFD) return bad("token stride smaller than head_dim");
  }
  if (reinterpret_cast<uintptr_t>(positions) & 3u) return bad("positions must be 4-byte aligned");
  if (reinterpret_cast<uintptr_t>(W) & 15u || reinterpret_cast<uintptr_t>(b) & 15u)
    return bad("W and b must be 16-byte aligned");

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  int dev = 0, sms = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess || (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) {
    set_error(std::string("kvx_fit_ridge: device query: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  kvx_ctx tmp;                       // for the RoPE tables only
  tmp.d = kFD;
  tmp.theta_s = cfg->src_rope_theta;
  tmp.theta_t = cfg->tgt_rope_theta;
  fill_rope(&tmp);

  FitParams P{};
  P.src = FitCache{static_cast<const __nv_bfloat16*>(src->k), static_cast<const __nv_bfloat16*>(src->v),
                   {src->stride[0], src->stride[1], src->stride[2], src->stride[3]}};
  P.tgt = FitCache{static_cast<const __nv_bfloat16*>(tgt->k), static_cast<const __nv_bfloat16*>(tgt->v),
                   {tgt->stride[0], tgt->stride[1], tgt->stride[2], tgt->stride[3]}};
  P.pos = positions;
  P.Ls = cfg->src_layers;
  P.Lt = cfg->tgt_layers;
  P.H = cfg->n_kv_heads;
  P.k = cfg->k;
  P.B = batch;
  P.T = tokens_per_seq;
  P.rope = tmp.rope;
  P.W = W;
  P.b = b;
  P.lambda = cfg->lambda;

  const int F = cfg->k * kFD;
  const size_t n_sys = static_cast<size_t>(cfg->tgt_layers) * 2 * cfg->n_kv_heads;
  const int Lmax = std::max(cfg->src_layers, cfg->tgt_layers);
  const size_t sums_n = static_cast<size_t>(2) * (cfg->src_layers + cfg->tgt_layers) * cfg->n_kv_heads * kFD;
  // the distinct (source layer, source layer) blocks of all target layers' Xc^T Xc
  const int kk = cfg->k;
  std::vector<int32_t> pair_list, pair_of(static_cast<size_t>(cfg->tgt_layers) * kk * kk, -1);
  {
    std::vector<int32_t> index(static_cast<size_t>(cfg->src_layers) * cfg->src_layers, -1);
    for (int l = 0; l < cfg->tgt_layers; ++l)
      for (int bi = 0; bi < kk; ++bi)
        for (int bj = 0; bj <= bi; ++bj) {
          int sa = cfg->selection[l * kk + bi], sb = cfg->selection[l * kk + bj];
          int ia = bi, ib = bj;
          if (sa < sb) {   // keep the block's rows on the larger layer; transpose in the solve
            std::swap(sa, sb);
            std::swap(ia, ib);
          }
          int32_t& idx = index[static_cast<size_t>(sa) * cfg->src_layers + sb];
          if (idx < 0) {
            idx = static_cast<int32_t>(pair_list.size() / 2);
            pair_list.push_back(sa);
            pair_list.push_back(sb);
          }
          pair_of[(static_cast<size_t>(l) * kk + bi) * kk + bj] = ia == bi ? idx : -1 - idx;
        }
  }
  const int n_pairs = static_cast<int>(pair_list.size() / 2);
  P.n_pairs = n_pairs;
  const size_t gram_n = static_cast<size_t>(2) * cfg->n_kv_heads * n_pairs * kFD * kFD;
  const size_t xty_n = n_sys * cfg->k * kFD * kFD;
  const int solve_grid = static_cast<int>(std::min<size_t>(n_sys, static_cast<size_t>(sms)));
  const size_t scratch_n = static_cast<size_t>(solve_grid) * (static_cast<size_t>(F) * F + static_cast<size_t>(F) * kFD);
  const size_t sel_n = static_cast<size_t>(cfg->tgt_layers) * cfg->k;
  std::vector<int32_t> tab(cfg->selection, cfg->selection + sel_n);
  tab.insert(tab.end(), pair_list.begin(), pair_list.end());
  tab.insert(tab.end(), pair_of.begin(), pair_of.end());
  const size_t bytes = sums_n * 8 + scratch_n * 8 + (gram_n + xty_n) * 4 + tab.size() * 4 + 16;
  char* ws = nullptr;
  if ((e = cudaMallocAsync(reinterpret_cast<void**>(&ws), bytes, st)) != cudaSuccess) {
    set_error(std::string("kvx_fit_ridge: workspace: ") + cudaGetErrorString(e));
    return KVX_ERR_OOM;
  }
  P.sums = reinterpret_cast<double*>(ws);
  P.scratch = P.sums + sums_n;
  P.gram = reinterpret_cast<float*>(P.scratch + scratch_n);
  P.xty = P.gram + gram_n;
  int32_t* dsel = reinterpret_cast<int32_t*>(P.xty + xty_n);
  P.sel = dsel;
  P.pairs = dsel + sel_n;
  P.pair_of = P.pairs + pair_list.size();
  P.status = dsel + tab.size();
  kvx_status result = KVX_OK;
  do {
    if ((e = cudaMemsetAsync(P.sums, 0, sums_n * 8, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(P.status, 0, 4, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(dsel, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice, st)) != cudaSuccess) {
      set_error(std::string("kvx_fit_ridge: setup: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    const int64_t N = static_cast<int64_t>(batch) * tokens_per_seq;
    const dim3 mgrid(static_cast<unsigned>((N + kFChunk - 1) / kFChunk), static_cast<unsigned>(4 * Lmax * cfg->n_kv_heads));
    fit_mean_kernel<<<mgrid, kFPairs, 0, st>>>(P, Lmax);
    const dim3 ggrid(static_cast<unsigned>(n_pairs + cfg->tgt_layers * kk), static_cast<unsigned>(2 * cfg->n_kv_heads));
    fit_gram_kernel<<<ggrid, 256, 0, st>>>(P);
    const size_t smem = static_cast<size_t>(kNB) * kNB * 8 + static_cast<size_t>(F - kNB) * kNB * 8;
    if ((e = cudaFuncSetAttribute(fit_solve_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem))) !=
        cudaSuccess) {
      set_error(std::string("kvx_fit_ridge: smem attribute: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    fit_solve_kernel<<<solve_grid, 256, smem, st>>>(P);
    if ((e = cudaGetLastError()) != cudaSuccess) {
      set_error(std::string("kvx_fit_ridge: launch: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    int32_t dstat = 0;
    if ((e = cudaMemcpyAsync(&dstat, P.status, 4, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess) {
      set_error(std::string("kvx_fit_ridge: run: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    if (dstat == kNotSpd) {
      set_error("kvx_fit_ridge: a system is not positive definite (lambda = 0 with too few tokens?)");
      result = KVX_ERR_INVALID_ARG;
    } else if (dstat != 0) {
      set_error("kvx_fit_ridge: a position is outside [0, 2^24)");
      result = static_cast<kvx_status>(dstat);
    }
  } while (false);
  cudaFreeAsync(ws, st);
  if (result == KVX_OK && (e = cudaStreamSynchronize(st)) != cudaSuccess) {
    set_error(std::string("kvx_fit_ridge: free: ") + cudaGetErrorString(e));
    result = KVX_ERR_CUDA;
  }
  return result;
}

}  // extern "C"
