// Ridge fit of the per-head mapper on the GPU (Sec. 3.1, Eq. Wstar; keys RoPE-stripped
// on both sides, Sec. 3.3).  For every target layer l, K|V and head h, over the N =
// B * T calibration tokens:
//   X = [x_{sel[l][0]} || ... || x_{sel[l][k-1]}]   (F = k d features; source keys with
//       the source RoPE stripped, source values as they are),
//   Y = head h of target layer l (target keys with the target RoPE stripped, values),
//   Xc, Yc centred by their column means,
//   W = (Xc^T Xc + lambda I)^{-1} Xc^T Yc,   b = mean(Y) - mean(X) W.
// bf16 caches, head_dim 128, half-split pairs.
// Cross-head mode (the paper's source feature, Appendix "Run information": d_s = k n_kv d):
// x_j is every KV head of layer sel[l][j] (head-minor), Y every head of target layer l, so
// there is one system per (l, K|V) with F = k H 128 features and H 128 right-hand sides:
// Xc^T Xc is formed and factored once per target layer and shared by its heads (Sec. 3.1).
//
// Steps:
// 1. Column sums and the centred Gram blocks on the tensor cores (kvx_gram.cu): a block
//    (source layer, source layer) of Xc^T Xc depends only on the two layers, K|V and the
//    head, so every distinct pair of the selection is computed once and shared by all
//    target layers whose selection holds both; the k blocks of Xc^T Yc are per target layer.
// 2. fit_solve_kernel: one CTA per system at a time (persistent); the block grid is
//    widened to float-float pairs (~48 significant bits, on the FP32 units) into a per-CTA
//    scratch matrix, lambda added, factorised by a blocked right-looking Cholesky (32-column
//    steps: the diagonal block factored by the CTA, its inverse, the panel as a product
//    with that inverse, the trailing update), then the two triangular solves for the d
//    right-hand sides in 32-row blocks (products with the solved rows, then the inverse
//    diagonal block) and the bias; W and b are written in fp32.
//    Cross-head systems: fit_solve_xh_kernel factorises one system per CTA (trailing
//    update staged per 128 x 128 tile), then fit_trisolve_xh_kernel solves and writes W and
//    b per (system, target head), so that the solves of fewer systems than SMs still fill
//    the GPU.
// kvx_fit_ridge runs them on the caller's stream, with stream-ordered workspace, and
// synchronises before it returns (the fit is an offline step).
#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <string>
#include <vector>

#include "kvx_gram.h"
#include "kvx_internal.h"
#include "kvx_ptx.cuh"

namespace kvx {
namespace {

using namespace ptx;

constexpr int kFD = 128;            // head_dim
constexpr int kNB = 32;             // Cholesky panel width
constexpr int64_t kMaxXhFeatures = 16384;   // cross-head F = k H 128 (2 GB of float-float matrix per CTA)

struct FitParams {
  const int32_t* sel;               // [L_t][k]
  int32_t Ls, Lt, H, k, B, T;
  double* sums;                     // [2 sides][2 kv][L][H][128]: side 0 L = L_s, side 1 L = L_t
  float* gram;                      // source-pair blocks: per head [2][H][n_pairs][128][128];
                                    // cross-head [n_pairs][2][H][H][128][128] (pair (sa, sb), blocks
                                    // (head of sa, head of sb); one layer: only row head >= column head)
  const int32_t* pairs;             // [n_pairs][2] source layers (sa >= sb)
  const int32_t* pair_of;           // [L_t][k][k] pair of block (bi, bj), bi >= bj
  int32_t n_pairs;
  float* xty;                       // per head [L_t][2][H][k][128][128]; cross-head
                                    // [L_t][2][k][H (source head)][H (target head)][128][128]
  double* scratch;                  // per CTA: F x F matrix + F x R right-hand sides + the F / 32
                                    // inverted 32 x 32 diagonal blocks of the factor
  float* W;                         // [L_t][2][H][F][128]
  float* b;                         // [L_t][2][H][128]
  double lambda;
  int32_t* status;
  int32_t R;                        // right-hand sides per system: 128 (per head) or H 128 (cross-head)
  int32_t sys0;                     // cross-head: first system of this launch (scratch slot = its offset)
};

__device__ __forceinline__ size_t sums_index(const FitParams& P, int side, int kv, int layer, int h) {
  const size_t base = side == 0 ? 0 : static_cast<size_t>(2) * P.Ls * P.H * kFD;
  const int L = side == 0 ? P.Ls : P.Lt;
  return base + ((static_cast<size_t>(kv) * L + layer) * P.H + h) * kFD;
}

__device__ __forceinline__ void report_fit(int32_t* status, int code) { atomicCAS(status, 0, code); }

// ------------------------------------------------------------------- solve --
// Float-float arithmetic: a value is the unevaluated sum hi + lo of two floats
// (|lo| <= ulp(hi) / 2), about 48 significant bits, against 53 for fp64 and far below the
// fp32 error of the Gram blocks it solves with.  GB300 runs 64 FP32 FMAs for each FP64 FMA,
// so the solve runs on the FP32 units: a fused multiply-add of two such pairs costs about a
// dozen FP32 instructions.  The error-free steps are the published ones: two_sum (Knuth,
// TAOCP vol. 2, 4.2.2), fast_two_sum (Dekker 1971, needs |a| >= |b|), two_prod by one
// FMA; the pair arithmetic follows Dekker's and the QD library's (Hida, Li, Bailey 2001)
// "sloppy" addition; the reciprocal square root of the pivots refines the hardware
// estimate by Newton's iteration (below).  The IEEE-rounded float divide and square root
// take several hundred cycles on the dependency chains of the factorisation, so pivots
// enter only through that reciprocal.
struct __align__(8) DF {
  float hi, lo;
};

__device__ __forceinline__ DF df_make(float a) { return DF{a, 0.f}; }
__device__ __forceinline__ DF fast_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return DF{s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ DF two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return DF{s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}
__device__ __forceinline__ DF df_neg(DF a) { return DF{-a.hi, -a.lo}; }
__device__ __forceinline__ DF df_add(DF a, DF b) {
  const DF s = two_sum(a.hi, b.hi);
  return fast_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(a.lo, b.lo)));
}
// a * b + c
__device__ __forceinline__ DF df_fma(DF a, DF b, DF c) {
  const float p = __fmul_rn(a.hi, b.hi);
  float e = __fmaf_rn(a.hi, b.hi, -p);
  e = __fmaf_rn(a.hi, b.lo, e);
  e = __fmaf_rn(a.lo, b.hi, e);
  const DF s = two_sum(p, c.hi);
  return fast_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(e, c.lo)));
}
// Dot-product accumulation with the renormalisation deferred: c.hi + c.lo is a running
// sum whose c.lo collects every step's rounding errors unnormalised (3 FP32 instructions
// fewer per step than df_fma); df_norm turns it back into a pair before the sum is used.
__device__ __forceinline__ DF df_fma_lazy(DF a, DF b, DF c) {
  const float p = __fmul_rn(a.hi, b.hi);
  float e = __fmaf_rn(a.hi, b.hi, -p);
  e = __fmaf_rn(a.hi, b.lo, e);
  e = __fmaf_rn(a.lo, b.hi, e);
  const DF s = two_sum(p, c.hi);
  return DF{s.hi, __fadd_rn(c.lo, __fadd_rn(s.lo, e))};
}
__device__ __forceinline__ DF df_norm(DF a) { return two_sum(a.hi, a.lo); }
__device__ __forceinline__ DF df_mul(DF a, DF b) {
  const float p = __fmul_rn(a.hi, b.hi);
  float e = __fmaf_rn(a.hi, b.hi, -p);
  e = __fmaf_rn(a.hi, b.lo, e);
  e = __fmaf_rn(a.lo, b.hi, e);
  return fast_two_sum(p, e);
}
__device__ __forceinline__ DF df_from_double(double x) {
  const float hi = static_cast<float>(x);
  return DF{hi, static_cast<float>(x - static_cast<double>(hi))};
}

// Persistent solve kernels: CTA c handles systems c, c + gridDim.x, ...  Dynamic shared
// memory holds pairs of floats (8 bytes an element, as fp64 was).
constexpr int kNotSpd = 100;        // internal status: a pivot <= 0 (matrix not positive definite)
constexpr int kPS = kNB + 1;        // panel row stride in shared memory (pairs)

constexpr int kSolveThreads = 512;                 // 16 warps: enough to keep the FP32 lanes busy

// 1 / sqrt(a), a > 0: y from the hardware estimate, then y += y (1 - a y^2) / 2 twice with
// the residual in float-float (Newton's iteration for the reciprocal square root, in the
// form of Karp and Markstein, ACM TOMS 23(4), 1997).
__device__ __forceinline__ DF df_rsqrt(DF a) {
  DF y = df_make(rsqrtf(a.hi));
#pragma unroll
  for (int it = 0; it < 2; ++it) {
    const DF r = df_fma(df_neg(a), df_mul(y, y), df_make(1.f));   // 1 - a y^2
    y = df_add(y, df_mul(y, df_make(__fmul_rn(0.5f, r.hi))));
  }
  return y;
}

// Shared-memory pieces of one factorisation step.
struct FactSmem {
  DF* D;        // [32][33]: the diagonal block, then its factor L_kk; D[i][32] = 1 / L[i][i]
  DF* X;        // [32][33]: L_kk^-1 (zeros above the diagonal)
  DF* Lc;       // [32]: the column of L formed in a step of the diagonal factorisation
  DF* T;        // [16][17]: scratch of the inverse
  DF* Pn;       // [pn_rows][33]: staged panel rows
  int pn_rows;
};
constexpr int kFactFixedDF = 2 * kNB * kPS + kNB + 16 * 17;   // D, X, Lc, T

// Cholesky of the 32 x 32 diagonal block at (c0, c0) of A (lower triangle) by the CTA:
// step j, warp 0 forms column j of L (the pivot through a float-float reciprocal square
// root), then every thread updates its entries (i, m), j < m <= i.  A pivot <= 0 is
// reported and its reciprocal square root taken as 1 so the call finishes.  Ends
// synchronised.
__device__ __forceinline__ void chol_diag(const DF* A, int F, int c0, const FactSmem& S, int32_t* status) {
  const int tid = threadIdx.x;
  DF* D = S.D;
  for (int e = tid; e < kNB * kNB; e += blockDim.x) {
    const int i = e / kNB, m = e % kNB;
    D[i * kPS + m] = m <= i ? A[static_cast<size_t>(c0 + i) * F + c0 + m] : df_make(0.f);
  }
  __syncthreads();
  for (int j = 0; j < kNB; ++j) {
    if (tid < kNB) {
      const DF d = D[j * kPS + j], own = D[tid * kPS + j];
      if (!(d.hi > 0.f) && tid == 0) report_fit(status, kNotSpd);
      const DF y = d.hi > 0.f ? df_rsqrt(d) : df_make(1.f);
      const DF l = tid > j ? df_mul(own, y) : (tid == j ? df_mul(d, y) : df_make(0.f));
      __syncwarp();
      S.Lc[tid] = l;
      if (tid >= j) D[tid * kPS + j] = l;
      if (tid == j) D[tid * kPS + kNB] = y;
    }
    __syncthreads();
    for (int e = tid; e < kNB * kNB; e += blockDim.x) {
      const int i = e / kNB, m = e % kNB;
      if (j < m && m <= i) D[i * kPS + m] = df_fma(df_neg(S.Lc[i]), S.Lc[m], D[i * kPS + m]);
    }
    __syncthreads();
  }
}

// X = L_kk^-1 by the CTA, for L = [[P, 0], [Q, R]] in 16 x 16 quarters: P^-1 and R^-1 by
// forward substitution (warps 0 and 1, lane = column), then the lower-left quarter
// -R^-1 (Q P^-1) as two 16 x 16 products; written row-major [32][32] to inv.  Ends
// synchronised.
__device__ __forceinline__ void tri_inverse(const FactSmem& S, DF* inv) {
  const int tid = threadIdx.x;
  const DF* D = S.D;
  DF* X = S.X;
  if (tid < 64 && (tid & 31) < 16) {
    const int o = 16 * (tid >> 5), j = tid & 31;
    for (int i = 0; i < 16; ++i) {
      DF v = df_make(i == j ? 1.f : 0.f);
      for (int m = j; m < i; ++m) v = df_fma_lazy(df_neg(D[(o + i) * kPS + o + m]), X[(o + m) * kPS + o + j], v);
      X[(o + i) * kPS + o + j] = i >= j ? df_mul(df_norm(v), D[(o + i) * kPS + kNB]) : df_make(0.f);
    }
  }
  for (int e = tid; e < 256; e += blockDim.x) X[(e / 16) * kPS + 16 + e % 16] = df_make(0.f);
  __syncthreads();
  if (tid < 256) {   // T = Q P^-1
    const int r = tid / 16, c = tid % 16;
    DF v = df_make(0.f);
    for (int m = c; m < 16; ++m) v = df_fma_lazy(D[(16 + r) * kPS + m], X[m * kPS + c], v);
    S.T[r * 17 + c] = df_norm(v);
  }
  __syncthreads();
  if (tid < 256) {   // lower-left quarter: -R^-1 T
    const int r = tid / 16, c = tid % 16;
    DF v = df_make(0.f);
    for (int m = 0; m <= r; ++m) v = df_fma_lazy(X[(16 + r) * kPS + 16 + m], S.T[m * 17 + c], v);
    X[(16 + r) * kPS + c] = df_neg(df_norm(v));
  }
  __syncthreads();
  for (int e = tid; e < kNB * kNB; e += blockDim.x) inv[e] = X[(e / kNB) * kPS + e % kNB];
}

// One 32-column step of the factorisation: the diagonal block and its inverse, then the
// panel X = A[c0 + 32 .., c0 .. c0 + 31] L_kk^-T, a product with the inverse (no dependency
// chains) computed from rows staged in S.Pn, S.pn_rows at a time, in 32-row tiles of 64
// threads x 4 x 4 entries, eight tiles per round; the result goes to A and, for the rows
// of the last chunk, stays in S.Pn (per-head systems stage every row in one chunk, so the
// trailing update reads the whole panel from there).  Ends synchronised.
__device__ __forceinline__ void chol_step(DF* A, int F, int c0, const FactSmem& S, DF* Inv, int32_t* status) {
  const int tid = threadIdx.x, rows = F - c0 - kNB;
  chol_diag(A, F, c0, S, status);
  tri_inverse(S, Inv + static_cast<size_t>(c0) * kNB);
  const int lt = tid & 63, ri = lt >> 3, cj = lt & 7;
  for (int r0 = 0; r0 < rows; r0 += S.pn_rows) {
    const int nr = min(S.pn_rows, rows - r0);
    for (int e = tid; e < nr * (kNB / 2); e += blockDim.x) {
      const int r = e / (kNB / 2), q = 2 * (e % (kNB / 2));
      const float4 v = *reinterpret_cast<const float4*>(A + static_cast<size_t>(c0 + kNB + r0 + r) * F + c0 + q);
      S.Pn[r * kPS + q] = DF{v.x, v.y};
      S.Pn[r * kPS + q + 1] = DF{v.z, v.w};
    }
    __syncthreads();
    const int tiles = (nr + kNB - 1) / kNB;
    for (int rd = 0; rd < tiles; rd += kSolveThreads / 64) {
      const int tile = rd + (tid >> 6);
      DF acc[4][4];
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = df_make(0.f);
      if (tile < tiles) {
        const DF* prow = S.Pn + (tile * kNB + ri) * kPS;
#pragma unroll 4
        for (int m = 0; m < kNB; ++m) {
          DF pi[4], pj[4];
#pragma unroll
          for (int a = 0; a < 4; ++a) pi[a] = prow[8 * a * kPS + m];
#pragma unroll
          for (int b = 0; b < 4; ++b) pj[b] = S.X[(cj + 8 * b) * kPS + m];
#pragma unroll
          for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[a][b] = df_fma_lazy(pi[a], pj[b], acc[a][b]);
        }
      }
      __syncthreads();   // the tile's rows are read before they are overwritten
      if (tile < tiles) {
#pragma unroll
        for (int a = 0; a < 4; ++a) {
          const int r = tile * kNB + ri + 8 * a;
          if (r >= nr) continue;
#pragma unroll
          for (int b = 0; b < 4; ++b) {
            const DF x = df_norm(acc[a][b]);
            S.Pn[r * kPS + cj + 8 * b] = x;
            A[static_cast<size_t>(c0 + kNB + r0 + r) * F + c0 + cj + 8 * b] = x;
          }
        }
      }
    }
    __syncthreads();
  }
}

// Asynchronous global -> shared copies (cp.async, completion tracked per thread by groups).
__device__ __forceinline__ void cp_async8(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

constexpr int kStageDF = kNB * kPS + kNB * kFD;   // one solve stage: [32][33] L entries + [32][128] rows
constexpr int kStages = 3;                         // solve stage buffers

// The two triangular solves with the factor L (lower triangle of A, leading dimension F)
// for 128 right-hand-side columns Z[0 .. F)[0 .. 128) (leading dimension ldz), in place:
// forward L Y = Z, then backward L^T W = Y, in 32-row blocks.  A block takes the products
// with the solved rows 32 at a time (chunk stages: 32 x 32 entries of L and 32 solved rows
// staged in shared memory; thread = 2 rows x 4 columns, 8 independent sums), then is
// multiplied by the inverse of its diagonal block (Inv, [F / 32][32][32], from the
// factorisation; its transpose in the backward solve), the same staged product with every
// thread busy.  Stages run through three shared-memory buffers: the next stage's operands
// are copied asynchronously while the current one computes, except where they are the
// rows the current stage solves (the chunk orders keep that to one stage per direction).
// fsm: kStages x kStageDF pairs.
__device__ __forceinline__ void tri_solves(const DF* A, int F, DF* Z, int ldz, const DF* Inv, DF* fsm) {
  const int tid = threadIdx.x;
  constexpr int kR = kNB * kFD / 4 / kSolveThreads;   // rows per thread (2)
  const int r0 = kR * (tid % (kNB / kR)), q0 = 4 * (tid / (kNB / kR));
  const int nb = F / kNB;
  auto load4 = [&](const DF* p, DF (&v)[4]) {
    const float4 x = *reinterpret_cast<const float4*>(p), y = *reinterpret_cast<const float4*>(p + 2);
    v[0] = DF{x.x, x.y};
    v[1] = DF{x.z, x.w};
    v[2] = DF{y.x, y.y};
    v[3] = DF{y.z, y.w};
  };
  // acc[a][c] -/+= sum_j Ls[r0 + a][j] Zs[j][q0 + c] (Ls indexed [row][j] when `rows_major`,
  // else [j][row])
  auto chunk_update = [&](const DF* Ls, const DF* Zs, DF (&acc)[kR][4], bool rows_major, bool subtract) {
#pragma unroll 4
    for (int j = 0; j < kNB; ++j) {
      DF z[4], l[kR];
      load4(&Zs[j * kFD + q0], z);
#pragma unroll
      for (int a2 = 0; a2 < kR; ++a2) {
        const DF v = rows_major ? Ls[(r0 + a2) * kPS + j] : Ls[j * kPS + r0 + a2];
        l[a2] = subtract ? df_neg(v) : v;
      }
#pragma unroll
      for (int a2 = 0; a2 < kR; ++a2)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a2][c] = df_fma_lazy(l[a2], z[c], acc[a2][c]);
    }
  };
  // Stage (bi, u) of one direction: block bi in solve order (b = bi forward, nb - 1 - bi
  // backward) has bi chunk stages u < bi, then its diagonal stage u = bi (mc < 0).  Chunk
  // rows: forward mc = u (ascending), backward mc = nb - 1 - u (descending).
  auto stage = [&](bool fwd, int bi, int u, int& b, int& mc) {
    b = fwd ? bi : nb - 1 - bi;
    mc = u == bi ? -1 : (fwd ? u : nb - 1 - u);
  };
  auto issue = [&](DF* buf, bool fwd, int b, int mc) {
    DF* Ls = buf;
    if (mc >= 0) {
      // forward: L[b + i][mc + j] -> Ls[i][j]; backward: L[mc + j][b + i] -> Ls[j][i]
      const int X = fwd ? b : mc, Y = fwd ? mc : b;
      for (int e = tid; e < kNB * kNB; e += blockDim.x)
        cp_async8(&Ls[(e / kNB) * kPS + e % kNB], &A[static_cast<size_t>(X * kNB + e / kNB) * F + Y * kNB + e % kNB]);
      float4* Zs = reinterpret_cast<float4*>(buf + kNB * kPS);
      for (int e = tid; e < kNB * kFD / 2; e += blockDim.x)
        cp_async16(&Zs[e], Z + static_cast<size_t>(mc * kNB + e / (kFD / 2)) * ldz + 2 * (e % (kFD / 2)));
    } else {
      const DF* inv = Inv + static_cast<size_t>(b) * kNB * kNB;
      for (int e = tid; e < kNB * kNB; e += blockDim.x) cp_async8(&Ls[(e / kNB) * kPS + e % kNB], &inv[e]);
    }
    cp_async_commit();
  };
  for (int dir = 0; dir < 2; ++dir) {
    const bool fwd = dir == 0;
    int bi = 0, u = 0, b = 0, mc = 0;
    stage(fwd, bi, u, b, mc);
    int k = 0;                                   // stages issued so far in this direction
    issue(fsm, fwd, b, mc);
    DF acc[kR][4];
#pragma unroll
    for (int a = 0; a < kR; ++a) load4(&Z[static_cast<size_t>(b * kNB + r0 + a) * ldz + q0], acc[a]);
    while (bi < nb) {
      DF* cur = fsm + (k % kStages) * kStageDF;
      DF* nxt = fsm + ((k + 1) % kStages) * kStageDF;
      const int bi2 = u < bi ? bi : bi + 1, u2 = u < bi ? u + 1 : 0;
      int b2 = 0, mc2 = 0;
      const bool more = bi2 < nb;
      if (more) stage(fwd, bi2, u2, b2, mc2);
      // the next stage's rows are the ones this diagonal stage solves: copy them after it
      const bool defer = more && mc < 0 && mc2 == b;
      if (more && !defer) {
        issue(nxt, fwd, b2, mc2);
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      __syncthreads();
      if (mc >= 0) {
        chunk_update(cur, cur + kNB * kPS, acc, fwd, true);
      } else {
        DF* Zs = cur + kNB * kPS;
#pragma unroll
        for (int a = 0; a < kR; ++a)
#pragma unroll
          for (int c = 0; c < 4; ++c) Zs[(r0 + a) * kFD + q0 + c] = df_norm(acc[a][c]);
        __syncthreads();
        DF res[kR][4];
#pragma unroll
        for (int a = 0; a < kR; ++a)
#pragma unroll
          for (int c = 0; c < 4; ++c) res[a][c] = df_make(0.f);
        chunk_update(cur, Zs, res, fwd, false);   // forward: L_kk^-1 [row][j]; backward: (L_kk^-1)^T
#pragma unroll
        for (int a = 0; a < kR; ++a)
#pragma unroll
          for (int c = 0; c < 4; ++c) Z[static_cast<size_t>(b * kNB + r0 + a) * ldz + q0 + c] = df_norm(res[a][c]);
      }
      // With three buffers the next issue targets the buffer of the stage two before this
      // one, which every thread left before the barrier above.  A diagonal stage ends with a
      // barrier: the next iteration issues its copies before its own barrier, and those may
      // read the rows this stage solved.
      if (mc < 0) {
        __syncthreads();
        if (defer) issue(nxt, fwd, b2, mc2);
      }
      if (more && mc < 0) {   // a new block starts: its right-hand sides
#pragma unroll
        for (int a = 0; a < kR; ++a) load4(&Z[static_cast<size_t>(b2 * kNB + r0 + a) * ldz + q0], acc[a]);
      }
      bi = bi2;
      u = u2;
      b = b2;
      mc = mc2;
      ++k;
    }
    __syncthreads();   // the direction's last stage is done with its buffer and its rows are written
  }
}

// b = mean(Y) - mean(X) W for one 128-column block of solved W (Z, leading dimension ldz),
// by the CTA in float-float: the F feature means (xmean(r), fp64 from the column sums)
// staged in shared memory as pairs, thread = (column tid % 128, quarter tid / 128 of the
// rows), the quarters' sums added in shared memory; ymean = this thread's column's mean of
// Y.  Writes b[0 .. 128) in fp32.  smem: F + 4 x 128 pairs.  Ends synchronised.
template <class XMean>
__device__ __forceinline__ void bias_out(int F, const DF* Z, int ldz, DF* smem, DF ymean, XMean xmean, float* b) {
  const int tid = threadIdx.x;
  constexpr int kQuarters = kSolveThreads / kFD;
  DF* xm = smem;
  DF* part = smem + F;
  for (int r = tid; r < F; r += blockDim.x) xm[r] = df_from_double(xmean(r));
  __syncthreads();
  const int c = tid % kFD, qtr = tid / kFD;
  DF acc = df_make(0.f);
  for (int r = qtr; r < F; r += kQuarters) acc = df_fma_lazy(xm[r], Z[static_cast<size_t>(r) * ldz + c], acc);
  part[qtr * kFD + c] = df_norm(acc);
  __syncthreads();
  if (tid < kFD) {
    DF v = ymean;
#pragma unroll
    for (int q = 0; q < kQuarters; ++q) v = df_add(v, df_neg(part[q * kFD + tid]));
    b[tid] = __fadd_rn(v.hi, v.lo);
  }
  __syncthreads();
}

// Per-head systems (F = 128 k <= 512): the whole panel stays in shared memory
// ([32][33] diagonal block + [F - 32][33] panel).
__global__ void __launch_bounds__(kSolveThreads, 1) fit_solve_kernel(const __grid_constant__ FitParams P) {
  extern __shared__ __align__(16) DF fsm[];
  // D, X, Lc, T, then the panel [F - 32][33] (rows padded so a warp's rows hit distinct banks)
  const FactSmem S{fsm, fsm + kNB * kPS, fsm + 2 * kNB * kPS, fsm + 2 * kNB * kPS + kNB, fsm + kFactFixedDF, 0};
  DF* Pn = S.Pn;
  const int F = P.k * kFD;
  const int tid = threadIdx.x;
  DF* A = reinterpret_cast<DF*>(P.scratch) +
          static_cast<size_t>(blockIdx.x) * (static_cast<size_t>(F) * F + static_cast<size_t>(F) * kFD +
                                             static_cast<size_t>(F) * kNB);
  DF* Z = A + static_cast<size_t>(F) * F;         // [F][128]
  DF* Inv = Z + static_cast<size_t>(F) * kFD;     // [F / 32][32][32]: inverses of the diagonal blocks
  const int n_sys = P.Lt * 2 * P.H;
  const double inv_n = 1.0 / (static_cast<double>(P.B) * P.T);
  const DF lam = df_from_double(P.lambda);
  for (int sys = blockIdx.x; sys < n_sys; sys += gridDim.x) {
    const int h = sys % P.H;
    const int kv = (sys / P.H) & 1;
    const int l = sys / (2 * P.H);
    // 1. A = Xc^T Xc + lambda I (the 128 x 128 blocks of the lower block triangle; the
    //    block of two selected layers is stored once per pair, transposed when the pair
    //    is) and Z = Xc^T Yc (contiguous per system); four entries per thread step
    for (int bi = 0; bi < P.k; ++bi) {
      for (int bj = 0; bj <= bi; ++bj) {
        const int pr = __ldg(&P.pair_of[(l * P.k + bi) * P.k + bj]);   // < 0: stored transposed
        const float* gb =
            P.gram + ((static_cast<size_t>(kv) * P.H + h) * P.n_pairs + (pr >= 0 ? pr : -1 - pr)) * kFD * kFD;
        for (int e = tid; e < kFD * kFD / 4; e += blockDim.x) {
          const int er = e / (kFD / 4), ec = 4 * (e % (kFD / 4));
          float g[4];
          if (pr >= 0) {
            const float4 v = *reinterpret_cast<const float4*>(gb + er * kFD + ec);
            g[0] = v.x;
            g[1] = v.y;
            g[2] = v.z;
            g[3] = v.w;
          } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) g[q] = gb[(ec + q) * kFD + er];
          }
          DF o[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) o[q] = bi == bj && er == ec + q ? df_add(df_make(g[q]), lam) : df_make(g[q]);
          float4* dst = reinterpret_cast<float4*>(A + static_cast<size_t>(bi * kFD + er) * F + bj * kFD + ec);
          dst[0] = make_float4(o[0].hi, o[0].lo, o[1].hi, o[1].lo);
          dst[1] = make_float4(o[2].hi, o[2].lo, o[3].hi, o[3].lo);
        }
      }
    }
    {
      const float4* xs = reinterpret_cast<const float4*>(P.xty + static_cast<size_t>(sys) * P.k * kFD * kFD);
      float4* zd = reinterpret_cast<float4*>(Z);
      for (int e = tid; e < F * kFD / 4; e += blockDim.x) {
        const float4 v = xs[e];
        zd[2 * e] = make_float4(v.x, 0.f, v.y, 0.f);
        zd[2 * e + 1] = make_float4(v.z, 0.f, v.w, 0.f);
      }
    }
    __syncthreads();
    // 2. Cholesky A = L L^T, lower triangle in place, 32-column panels
    for (int c0 = 0; c0 < F; c0 += kNB) {
      FactSmem Sp = S;
      Sp.pn_rows = F - c0 - kNB > 0 ? F - c0 - kNB : 1;
      chol_step(A, F, c0, Sp, Inv, P.status);
      // trailing update: A[i][j] -= P[i] . P[j] for c0+32 <= j <= i, in 32 x 32 tiles of the
      // lower triangle, eight at a time; a tile is 64 threads of 4 x 4 entries (rows ri + 8a,
      // columns cj + 8b: a warp's panel loads hit distinct banks), A's entries loaded first
      const int rows = F - c0 - kNB;
      const int nt = rows / kNB;
      const int lt = tid & 63, ri = lt >> 3, cj = lt & 7;
      for (int tile = tid >> 6; tile < nt * (nt + 1) / 2; tile += kSolveThreads / 64) {
        int ti = 0;
        while ((ti + 1) * (ti + 2) / 2 <= tile) ++ti;
        const int tj = tile - ti * (ti + 1) / 2;
        const int gi = ti * kNB + ri, gj = tj * kNB + cj;
        DF acc[4][4], aold[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b) {
            acc[a][b] = df_make(0.f);
            aold[a][b] = gj + 8 * b <= gi + 8 * a ? A[static_cast<size_t>(c0 + kNB + gi + 8 * a) * F + c0 + kNB + gj + 8 * b]
                                                  : df_make(0.f);
          }
#pragma unroll 4
        for (int m = 0; m < kNB; ++m) {
          DF pi[4], pj[4];
#pragma unroll
          for (int a = 0; a < 4; ++a) pi[a] = Pn[(gi + 8 * a) * kPS + m];
#pragma unroll
          for (int b = 0; b < 4; ++b) pj[b] = Pn[(gj + 8 * b) * kPS + m];
#pragma unroll
          for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[a][b] = df_fma_lazy(pi[a], pj[b], acc[a][b]);
        }
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b)
            if (gj + 8 * b <= gi + 8 * a)
              A[static_cast<size_t>(c0 + kNB + gi + 8 * a) * F + c0 + kNB + gj + 8 * b] =
                  df_add(aold[a][b], df_neg(df_norm(acc[a][b])));
      }
      __syncthreads();
    }
    // 3. forward and backward solves for the 128 right-hand sides
    tri_solves(A, F, Z, kFD, Inv, fsm);
    // 4. W (fp32) and b = mean(Y) - mean(X) W
    float* Wout = P.W + static_cast<size_t>(sys) * F * kFD;
    for (int64_t e = tid; e < static_cast<int64_t>(F) * kFD; e += blockDim.x) Wout[e] = __fadd_rn(Z[e].hi, Z[e].lo);
    bias_out(
        F, Z, kFD, fsm, df_from_double(P.sums[sums_index(P, 1, kv, l, h) + (tid & (kFD - 1))] * inv_n),
        [&](int r) { return P.sums[sums_index(P, 0, kv, __ldg(&P.sel[l * P.k + r / kFD]), h) + r % kFD] * inv_n; },
        P.b + static_cast<size_t>(sys) * kFD);
  }
}

// Cross-head systems (Sec. 3.1 with the source feature of Appendix "Run information":
// d_s = k n_kv d): one system per (target layer, K|V), F = k H 128 features (selected
// layer-major, head-minor), R = H 128 right-hand sides (every target head of the layer),
// so X_c^T X_c is formed and factored once per target layer and shared by its heads.
// The matrix is too large for the panel to stay in shared memory: the trailing update
// runs in 128 x 128 tiles whose two 128-row panel slices are staged per tile.  One system
// per CTA and launch (scratch slot = blockIdx.x); fit_trisolve_xh_kernel then solves.
constexpr int kXT = 128;                          // trailing-update tile
constexpr int kXPanelRows = 512;                  // panel rows staged at a time
static_assert(4 * kXT <= kXPanelRows, "the trailing update's two buffers of panel slices take the panel chunk's place");
__global__ void __launch_bounds__(kSolveThreads, 1) fit_solve_xh_kernel(const __grid_constant__ FitParams P) {
  extern __shared__ __align__(16) DF fsm[];
  // D, X, Lc, T, then a chunk of panel rows [kXPanelRows][33]; the trailing update's two
  // buffers of panel slices ([2][128][33] each) take the chunk's place
  const FactSmem S{fsm, fsm + kNB * kPS, fsm + 2 * kNB * kPS, fsm + 2 * kNB * kPS + kNB, fsm + kFactFixedDF, kXPanelRows};
  const int H = P.H, R = P.R;
  const int F = P.k * H * kFD;
  const int tid = threadIdx.x;
  DF* A = reinterpret_cast<DF*>(P.scratch) +
          static_cast<size_t>(blockIdx.x) * (static_cast<size_t>(F) * F + static_cast<size_t>(F) * R +
                                             static_cast<size_t>(F) * kNB);
  DF* Z = A + static_cast<size_t>(F) * F;         // [F][R]
  DF* Inv = Z + static_cast<size_t>(F) * R;       // [F / 32][32][32]: inverses of the diagonal blocks
  const int n_sys = P.Lt * 2;
  const DF lam = df_from_double(P.lambda);
  constexpr size_t kBlk = static_cast<size_t>(kFD) * kFD;
  {
    const int sys = P.sys0 + static_cast<int>(blockIdx.x);
    if (sys >= n_sys) return;
    const int kv = sys & 1;
    const int l = sys >> 1;
    // 1. A = Xc^T Xc + lambda I (lower triangle) from the source-pair blocks, Z = Xc^T Yc
    for (int64_t e = tid; e < static_cast<int64_t>(F) * F; e += blockDim.x) {
      const int r = static_cast<int>(e / F), c = static_cast<int>(e % F);
      if (c > r) continue;
      const int ur = r / kFD, uc = c / kFD;       // feature blocks (layer j, head x), ur >= uc
      const int bi = ur / H, bj = uc / H;
      int hr = ur % H, hc = uc % H, er = r % kFD, ec = c % kFD;
      const int pr = __ldg(&P.pair_of[(l * P.k + bi) * P.k + bj]);
      const int q = pr >= 0 ? pr : -1 - pr;
      if (pr < 0) {                               // stored as (sel[bj], sel[bi]): transpose
        const int t = hr; hr = hc; hc = t;
        const int u = er; er = ec; ec = u;
      }
      if (hr < hc && __ldg(&P.pairs[2 * q]) == __ldg(&P.pairs[2 * q + 1])) {   // one layer: only hr >= hc stored
        const int t = hr; hr = hc; hc = t;
        const int u = er; er = ec; ec = u;
      }
      const float g = P.gram[(((static_cast<size_t>(q) * 2 + kv) * H + hr) * H + hc) * kBlk +
                             static_cast<size_t>(er) * kFD + ec];
      A[e] = r == c ? df_add(df_make(g), lam) : df_make(g);
    }
    for (int64_t e = tid; e < static_cast<int64_t>(F) * R; e += blockDim.x) {
      const int r = static_cast<int>(e / R), col = static_cast<int>(e % R);
      const int u = r / kFD, ht = col / kFD;      // u = bi * H + x
      Z[e] = df_make(P.xty[((((static_cast<size_t>(l) * 2 + kv) * P.k * H + u) * H + ht)) * kBlk +
                           static_cast<size_t>(r % kFD) * kFD + col % kFD]);
    }
    __syncthreads();
    // 2. Cholesky, 32-column panels; trailing update in 128 x 128 tiles of the lower triangle
    for (int c0 = 0; c0 < F; c0 += kNB) {
      chol_step(A, F, c0, S, Inv, P.status);
      // trailing update in 128 x 128 tiles of the lower triangle: the tile's two 128-row
      // slices of the panel staged in shared memory by cp.async, the next tile's while this
      // one computes (two buffers); thread = 8 rows (ri + 16a) x 4 columns (cj + 32b), so a
      // warp's row loads are broadcasts; the sums start from A's entries (loaded while the
      // slices land) and are written back without a wait
      const int base = c0 + kNB, rows = F - base;
      const int nt = (rows + kXT - 1) / kXT, ntiles = nt * (nt + 1) / 2;
      const int ri = tid >> 5, cj = tid & 31;
      auto tile_ij = [](int tile, int& ti, int& tj) {
        ti = 0;
        while ((ti + 1) * (ti + 2) / 2 <= tile) ++ti;
        tj = tile - ti * (ti + 1) / 2;
      };
      auto issue_slices = [&](int tile, DF* dst) {
        int ti, tj;
        tile_ij(tile, ti, tj);
        for (int e = tid; e < 2 * kXT * kNB; e += blockDim.x) {
          const int sl = e / (kXT * kNB), rr = (e / kNB) % kXT, m = e % kNB;
          const int row = (sl == 0 ? ti : tj) * kXT + rr;
          DF* d = dst + (sl * kXT + rr) * kPS + m;
          if (row < rows) cp_async8(d, A + static_cast<size_t>(base + row) * F + c0 + m);
          else *d = df_make(0.f);
        }
        cp_async_commit();
      };
      if (ntiles > 0) issue_slices(0, S.Pn);
      for (int tile = 0; tile < ntiles; ++tile) {
        int ti, tj;
        tile_ij(tile, ti, tj);
        if (tile + 1 < ntiles) issue_slices(tile + 1, S.Pn + ((tile + 1) & 1) * 2 * kXT * kPS);
        // this thread's entries: rows gi0 + 16a, columns gj0 + 32b of the trailing block
        const int gi0 = ti * kXT + ri, gj0 = tj * kXT + cj;
        DF* const a0 = A + static_cast<size_t>(base + gi0) * F + base + gj0;
        const size_t row16 = static_cast<size_t>(16) * F;
        DF acc[8][4];
#pragma unroll
        for (int a = 0; a < 8; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b)
            acc[a][b] = gi0 + 16 * a < rows && gj0 + 32 * b <= gi0 + 16 * a ? a0[a * row16 + 32 * b] : df_make(0.f);
        if (tile + 1 < ntiles) cp_async_wait<1>();
        else cp_async_wait<0>();
        __syncthreads();
        const DF* Pi = S.Pn + (tile & 1) * 2 * kXT * kPS;
        const DF* Pj = Pi + kXT * kPS;
#pragma unroll 2
        for (int m = 0; m < kNB; ++m) {
          DF pi[8], pj[4];
#pragma unroll
          for (int a = 0; a < 8; ++a) pi[a] = Pi[(ri + 16 * a) * kPS + m];
#pragma unroll
          for (int b = 0; b < 4; ++b) pj[b] = Pj[(cj + 32 * b) * kPS + m];
#pragma unroll
          for (int a = 0; a < 8; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[a][b] = df_fma_lazy(df_neg(pi[a]), pj[b], acc[a][b]);
        }
#pragma unroll
        for (int a = 0; a < 8; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b)
            if (gi0 + 16 * a < rows && gj0 + 32 * b <= gi0 + 16 * a) a0[a * row16 + 32 * b] = df_norm(acc[a][b]);
        __syncthreads();   // the buffer is free for the slices of tile + 2
      }
    }
  }
}

// Cross-head triangular solves and outputs, one unit per (system of the launch, target
// head): the factor, its inverted diagonal blocks and the right-hand sides come from the
// scratch slot that fit_solve_xh_kernel factored, and the H units of a system run on
// different SMs (the factorisation occupies one SM per system; there are often fewer
// systems than SMs).
__global__ void __launch_bounds__(kSolveThreads, 1) fit_trisolve_xh_kernel(const __grid_constant__ FitParams P,
                                                                           int n_slots) {
  extern __shared__ __align__(16) DF fsm[];
  const int H = P.H, R = P.R;
  const int F = P.k * H * kFD;
  const int tid = threadIdx.x;
  const double inv_n = 1.0 / (static_cast<double>(P.B) * P.T);
  const int n_units = n_slots * H;
  for (int u = blockIdx.x; u < n_units; u += gridDim.x) {
    const int slot = u / H, ht = u % H;
    const int sys = P.sys0 + slot;
    const int kv = sys & 1, l = sys >> 1;
    DF* A = reinterpret_cast<DF*>(P.scratch) +
            static_cast<size_t>(slot) * (static_cast<size_t>(F) * F + static_cast<size_t>(F) * R +
                                         static_cast<size_t>(F) * kNB);
    DF* Z = A + static_cast<size_t>(F) * F;
    const DF* Inv = Z + static_cast<size_t>(F) * R;
    DF* Zh = Z + static_cast<size_t>(ht) * kFD;   // this head's 128 columns, leading dimension R
    tri_solves(A, F, Zh, R, Inv, fsm);
    // W (fp32, [L_t][2][H][F][128]) and b = mean(Y) - mean(X) W of target head ht
    float* Wout = P.W + (static_cast<size_t>(sys) * H + ht) * F * kFD;
    for (int64_t e = tid; e < static_cast<int64_t>(F) * kFD; e += blockDim.x) {
      const int r = static_cast<int>(e / kFD), c = static_cast<int>(e % kFD);
      const DF z = Zh[static_cast<size_t>(r) * R + c];
      Wout[e] = __fadd_rn(z.hi, z.lo);
    }
    bias_out(
        F, Zh, R, fsm, df_from_double(P.sums[sums_index(P, 1, kv, l, ht) + (tid & (kFD - 1))] * inv_n),
        [&](int r) {
          const int uu = r / kFD;
          return P.sums[sums_index(P, 0, kv, __ldg(&P.sel[l * P.k + uu / H]), uu % H) + r % kFD] * inv_n;
        },
        P.b + (static_cast<size_t>(sys) * H + ht) * kFD);
  }
}

// Host plan of a fit: the distinct source pairs, the block tables, the operand slots and
// the sizes of every device piece (the same for the run and the workspace query).
struct FitPlan {
  std::vector<int32_t> pair_list, pair_of, tab, slot_of_src;
  int n_pairs = 0, solve_grid = 0, F = 0, R = 0;
  bool cross = false;
  size_t n_sys = 0, sums_n = 0, gram_n = 0, xty_n = 0, scratch_n = 0, sel_n = 0, n_blocks = 0;
  size_t fixed_bytes = 0;          // sums, scratch, blocks, tables, status (256-aligned pieces)
};

size_t al256(size_t n) { return (n + 255) / 256 * 256; }

// Bytes of per-CTA solve scratch the cross-head fit may take (the grid shrinks beyond it).
constexpr size_t kXhScratchCap = static_cast<size_t>(80) << 30;

FitPlan plan_fit(const kvx_fit_config* cfg, int sms, GramSpec* G) {
  FitPlan p;
  const int kk = cfg->k;
  const bool cross = cfg->head_mix == KVX_CROSS_HEAD;
  const int H = cfg->n_kv_heads;
  p.cross = cross;
  p.F = kk * kFD * (cross ? H : 1);
  p.R = cross ? H * kFD : kFD;
  p.n_sys = static_cast<size_t>(cfg->tgt_layers) * 2 * (cross ? 1 : H);
  p.sums_n = static_cast<size_t>(2) * (cfg->src_layers + cfg->tgt_layers) * cfg->n_kv_heads * kFD;
  p.pair_of.assign(static_cast<size_t>(cfg->tgt_layers) * kk * kk, -1);
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
          idx = static_cast<int32_t>(p.pair_list.size() / 2);
          p.pair_list.push_back(sa);
          p.pair_list.push_back(sb);
        }
        p.pair_of[(static_cast<size_t>(l) * kk + bi) * kk + bj] = ia == bi ? idx : -1 - idx;
      }
  p.n_pairs = static_cast<int>(p.pair_list.size() / 2);
  const size_t kBlk = static_cast<size_t>(kFD) * kFD;
  p.gram_n = static_cast<size_t>(2) * H * (cross ? H : 1) * p.n_pairs * kBlk;
  p.xty_n = static_cast<size_t>(cfg->tgt_layers) * 2 * H * kk * (cross ? H : 1) * kBlk;
  p.solve_grid = static_cast<int>(std::min<size_t>(p.n_sys, static_cast<size_t>(std::max(sms, 1))));
  const size_t per_cta = static_cast<size_t>(p.F) * p.F + static_cast<size_t>(p.F) * p.R + static_cast<size_t>(p.F) * kNB;
  if (cross)
    p.solve_grid = static_cast<int>(std::max<size_t>(1, std::min<size_t>(p.solve_grid, kXhScratchCap / (per_cta * 8))));
  p.scratch_n = static_cast<size_t>(p.solve_grid) * per_cta;
  p.sel_n = static_cast<size_t>(cfg->tgt_layers) * kk;
  p.tab.assign(cfg->selection, cfg->selection + p.sel_n);
  p.tab.insert(p.tab.end(), p.pair_list.begin(), p.pair_list.end());
  p.tab.insert(p.tab.end(), p.pair_of.begin(), p.pair_of.end());
  // operands: the selected source layers, then every target layer
  p.slot_of_src.assign(cfg->src_layers, -1);
  for (size_t i = 0; i < p.sel_n; ++i) p.slot_of_src[cfg->selection[i]] = 0;
  G->slot_side.clear();
  G->slot_layer.clear();
  for (int L = 0; L < cfg->src_layers; ++L)
    if (p.slot_of_src[L] == 0) {
      p.slot_of_src[L] = static_cast<int32_t>(G->slot_side.size());
      G->slot_side.push_back(0);
      G->slot_layer.push_back(L);
    }
  for (int l = 0; l < cfg->tgt_layers; ++l) {
    G->slot_side.push_back(1);
    G->slot_layer.push_back(l);
  }
  G->H = cfg->n_kv_heads;
  if (cross) {   // per (pair, K|V): H x H head blocks (one layer: row head >= column head); cross: k H H per (l, K|V)
    size_t nb = 0;
    for (int q = 0; q < p.n_pairs; ++q) nb += p.pair_list[2 * q] == p.pair_list[2 * q + 1] ? H * (H + 1) / 2 : H * H;
    p.n_blocks = 2 * nb + static_cast<size_t>(2) * cfg->tgt_layers * kk * H * H;
  } else {
    p.n_blocks = static_cast<size_t>(2) * cfg->n_kv_heads * (p.n_pairs + p.sel_n);
  }
  p.fixed_bytes = al256(p.sums_n * 8) + al256(p.scratch_n * 8) + al256((p.gram_n + p.xty_n) * 4) +
                  al256(p.tab.size() * 4 + 4) + gram_fixed_bytes(*G, p.n_blocks);
  return p;
}

const char* check_fit_config(const kvx_fit_config* cfg) {
  if (!cfg) return "NULL argument";
  if (cfg->head_dim != kFD) return "head_dim must be 128";
  if (cfg->head_mix != KVX_PER_HEAD && cfg->head_mix != KVX_CROSS_HEAD) return "bad head_mix";
  if (cfg->head_mix == KVX_PER_HEAD && (cfg->k < 1 || cfg->k > 4)) return "k must be in [1, 4] (per head)";
  if (cfg->head_mix == KVX_CROSS_HEAD &&
      (cfg->k < 1 || static_cast<int64_t>(cfg->k) * cfg->n_kv_heads * kFD > kMaxXhFeatures))
    return "k * n_kv_heads * 128 must be in [128, 16384] (cross-head)";
  if (cfg->src_layers < 1 || cfg->tgt_layers < 1 || cfg->n_kv_heads < 1 || cfg->k > cfg->src_layers)
    return "layer / head counts out of range";
  if (!(cfg->lambda >= 0.0) || !(cfg->src_rope_theta > 1.0) || !(cfg->tgt_rope_theta > 1.0))
    return "lambda must be >= 0 and the RoPE bases > 1";
  if (!cfg->selection) return "NULL selection";
  for (int64_t i = 0; i < static_cast<int64_t>(cfg->tgt_layers) * cfg->k; ++i)
    if (cfg->selection[i] < 0 || cfg->selection[i] >= cfg->src_layers) return "selection entry out of range";
  if (cfg->workspace_bytes != 0 && !cfg->workspace) return "workspace_bytes without a workspace";
  if (cfg->rope_numerics != KVX_ROPE_EXACT && cfg->rope_numerics != KVX_ROPE_HF) return "bad rope_numerics";
  if (const char* why = check_rope_scaling(cfg->src_rope_scaling)) return why;
  if (const char* why = check_rope_scaling(cfg->tgt_rope_scaling)) return why;
  if (reinterpret_cast<uintptr_t>(cfg->workspace) & 255u) return "workspace must be 256-byte aligned";
  return nullptr;
}

int sm_count_or_zero() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return sms;
}

}  // namespace
}  // namespace kvx

extern "C" {

KVX_API int64_t kvx_fit_workspace_bytes(const kvx_fit_config* cfg, int32_t batch, int32_t tokens_per_seq) {
  using namespace kvx;
  if (check_fit_config(cfg) || batch < 1 || tokens_per_seq < 1) return -1;
  const int sms = sm_count_or_zero();
  if (sms <= 0) return -1;
  GramSpec G;
  const FitPlan p = plan_fit(cfg, sms, &G);
  const int64_t N = static_cast<int64_t>(batch) * tokens_per_seq;
  const size_t np = static_cast<size_t>((N + 63) / 64 * 64);
  return static_cast<int64_t>(p.fixed_bytes + gram_bytes_per_token(G) * np + 1024);
}

KVX_API kvx_status kvx_fit_ridge(const kvx_fit_config* cfg, const kvx_src* src, const kvx_src* tgt, int32_t batch,
                                 int32_t tokens_per_seq, const int32_t* positions, float* W, float* b,
                                 void* stream) {
  using namespace kvx;
  NvtxRange range("kvx_fit_ridge");
  set_error("");
  auto bad = [](const char* m) {
    set_error(std::string("kvx_fit_ridge: ") + m);
    return KVX_ERR_INVALID_ARG;
  };
  if (const char* why = check_fit_config(cfg)) return bad(why);
  if (!src || !tgt || !positions || !W || !b) return bad("NULL argument");
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
  const int sms = sm_count_or_zero();
  if (sms <= 0) {
    set_error("kvx_fit_ridge: device query failed");
    return KVX_ERR_CUDA;
  }
  kvx_ctx tmp;                       // for the RoPE tables only
  tmp.d = kFD;
  tmp.theta_s = cfg->src_rope_theta;
  tmp.theta_t = cfg->tgt_rope_theta;
  set_rope_scaling(&tmp, cfg->src_rope_scaling, cfg->tgt_rope_scaling);
  fill_rope(&tmp);

  GramSpec G;
  const FitPlan pl = plan_fit(cfg, sms, &G);
  G.cache[0] = GramCache{src->k, src->v, {src->stride[0], src->stride[1], src->stride[2], src->stride[3]}};
  G.cache[1] = GramCache{tgt->k, tgt->v, {tgt->stride[0], tgt->stride[1], tgt->stride[2], tgt->stride[3]}};
  G.pos = positions;
  G.B = batch;
  G.T = tokens_per_seq;
  G.Ls = cfg->src_layers;
  G.Lt = cfg->tgt_layers;
  G.rope = tmp.rope;
  G.hf = cfg->rope_numerics == KVX_ROPE_HF;
  G.sm_count = sms;

  // device pieces: from the caller's workspace, or one stream-ordered allocation
  Scratch S;
  char* own = nullptr;
  const bool caller_ws = cfg->workspace != nullptr;
  const size_t fit_bytes = pl.fixed_bytes - gram_fixed_bytes(G, pl.n_blocks);
  if (caller_ws) {
    S.p = static_cast<char*>(cfg->workspace);
    S.bytes = static_cast<size_t>(cfg->workspace_bytes);
    if (S.bytes < pl.fixed_bytes) return bad("workspace too small (see kvx_fit_workspace_bytes)");
  } else {
    if ((e = cudaMallocAsync(reinterpret_cast<void**>(&own), fit_bytes, st)) != cudaSuccess) {
      set_error(std::string("kvx_fit_ridge: workspace: ") + cudaGetErrorString(e));
      return KVX_ERR_OOM;
    }
    S.p = own;
    S.bytes = fit_bytes;
  }
  FitParams P{};
  P.Ls = cfg->src_layers;
  P.Lt = cfg->tgt_layers;
  P.H = cfg->n_kv_heads;
  P.k = cfg->k;
  P.B = batch;
  P.T = tokens_per_seq;
  P.W = W;
  P.b = b;
  P.lambda = cfg->lambda;
  P.R = pl.R;
  P.n_pairs = pl.n_pairs;
  P.sums = reinterpret_cast<double*>(S.take(pl.sums_n * 8));
  P.scratch = reinterpret_cast<double*>(S.take(pl.scratch_n * 8));
  P.gram = reinterpret_cast<float*>(S.take((pl.gram_n + pl.xty_n) * 4));
  P.xty = P.gram + pl.gram_n;
  int32_t* dsel = reinterpret_cast<int32_t*>(S.take(pl.tab.size() * 4 + 4));
  P.sel = dsel;
  P.pairs = dsel + pl.sel_n;
  P.pair_of = P.pairs + pl.pair_list.size();
  P.status = dsel + pl.tab.size();
  if (!caller_ws) S = Scratch{};     // the Gram engine allocates its own
  kvx_status result = KVX_OK;
  PhaseTimer timer(st);
  do {
    if ((e = cudaMemsetAsync(P.sums, 0, pl.sums_n * 8, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(P.status, 0, 4, st)) != cudaSuccess ||
        (e = cudaMemcpyAsync(dsel, pl.tab.data(), pl.tab.size() * 4, cudaMemcpyHostToDevice, st)) != cudaSuccess) {
      set_error(std::string("kvx_fit_ridge: setup: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    G.sums = P.sums;
    G.status = P.status;
    const int kk = cfg->k;
    const int32_t tslot0 = static_cast<int32_t>(G.slot_side.size()) - cfg->tgt_layers;
    std::vector<GramBlock> blocks;
    blocks.reserve(pl.n_blocks);
    const int H = cfg->n_kv_heads;
    const size_t kBlk = static_cast<size_t>(kFD) * kFD;
    if (pl.cross) {
      for (int q = 0; q < pl.n_pairs; ++q) {
        const int sa = pl.pair_list[2 * q], sb = pl.pair_list[2 * q + 1];
        for (int kv = 0; kv < 2; ++kv)
          for (int x = 0; x < H; ++x)
            for (int y = 0; y < H; ++y) {
              if (sa == sb && x < y) continue;
              GramBlock g{pl.slot_of_src[sa], pl.slot_of_src[sb], kv, x,
                          P.gram + (((static_cast<size_t>(q) * 2 + kv) * H + x) * H + y) * kBlk};
              g.hb = y;
              blocks.push_back(g);
            }
      }
      for (int l = 0; l < cfg->tgt_layers; ++l)
        for (int kv = 0; kv < 2; ++kv)
          for (int bi = 0; bi < kk; ++bi)
            for (int x = 0; x < H; ++x)
              for (int ht = 0; ht < H; ++ht) {
                GramBlock g{pl.slot_of_src[cfg->selection[l * kk + bi]], tslot0 + l, kv, x,
                            P.xty + ((((static_cast<size_t>(l) * 2 + kv) * kk + bi) * H + x) * H + ht) * kBlk};
                g.hb = ht;
                blocks.push_back(g);
              }
    }
    for (int kv = 0; kv < 2 && !pl.cross; ++kv)
      for (int h = 0; h < cfg->n_kv_heads; ++h) {
        for (int q = 0; q < pl.n_pairs; ++q)
          blocks.push_back(GramBlock{pl.slot_of_src[pl.pair_list[2 * q]], pl.slot_of_src[pl.pair_list[2 * q + 1]], kv,
                                     h, P.gram + ((static_cast<size_t>(kv) * cfg->n_kv_heads + h) * pl.n_pairs + q) *
                                                     kFD * kFD});
        for (int l = 0; l < cfg->tgt_layers; ++l)
          for (int bi = 0; bi < kk; ++bi)
            blocks.push_back(GramBlock{pl.slot_of_src[cfg->selection[l * kk + bi]], tslot0 + l, kv, h,
                                       P.xty + (((static_cast<size_t>(l) * 2 + kv) * cfg->n_kv_heads + h) * kk + bi) *
                                                   kFD * kFD});
      }
    size_t budget = 0;
    if (!caller_ws) {
      size_t free_b = 0, total_b = 0;
      if ((e = cudaMemGetInfo(&free_b, &total_b)) != cudaSuccess) {
        set_error(std::string("kvx_fit_ridge: memory query: ") + cudaGetErrorString(e));
        result = KVX_ERR_CUDA;
        break;
      }
      budget = std::min<size_t>(free_b / 2, static_cast<size_t>(32) << 30);
    }
    Scratch* sp = caller_ws ? &S : nullptr;
    if ((result = gram_sums(G, st, &timer, sp)) != KVX_OK ||
        (result = gram_blocks(G, blocks, budget, st, &timer, sp)) != KVX_OK) {
      set_error(std::string("kvx_fit_ridge: ") + kvx_last_error());
      break;
    }
    // the factorisation's diagonal block and panel (per head) or tile slices (cross-head),
    // or the solves' staged chunk
    const size_t fact = kFactFixedDF + static_cast<size_t>(pl.cross ? kXPanelRows : pl.F - kNB) * kPS;
    const size_t smem = std::max(fact, static_cast<size_t>(kStages) * kStageDF) * 8;
    auto kernel = pl.cross ? fit_solve_xh_kernel : fit_solve_kernel;
    if ((e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem))) !=
            cudaSuccess ||
        (pl.cross && (e = cudaFuncSetAttribute(fit_trisolve_xh_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(smem))) != cudaSuccess)) {
      set_error(std::string("kvx_fit_ridge: smem attribute: ") + cudaGetErrorString(e));
      result = KVX_ERR_CUDA;
      break;
    }
    timer.begin(3);
    if (!pl.cross) {
      kernel<<<pl.solve_grid, kSolveThreads, smem, st>>>(P);
    } else {
      // waves of solve_grid systems (the scratch holds that many factors): factorise, then
      // the triangular solves of the wave's systems, one unit per (system, target head)
      const int n_sys = static_cast<int>(pl.n_sys);
      for (int s0 = 0; s0 < n_sys; s0 += pl.solve_grid) {
        P.sys0 = s0;
        const int slots = std::min(pl.solve_grid, n_sys - s0);
        fit_solve_xh_kernel<<<slots, kSolveThreads, smem, st>>>(P);
        const int units = slots * static_cast<int>(cfg->n_kv_heads);
        fit_trisolve_xh_kernel<<<std::min(units, std::max(sms, 1)), kSolveThreads, smem, st>>>(P, slots);
      }
    }
    timer.end();
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
    } else if (dstat == KVX_ERR_DEVICE_BOUNDS) {
      set_error("kvx_fit_ridge: a position is outside [0, 2^24)");
      result = KVX_ERR_DEVICE_BOUNDS;
    } else if (dstat != 0) {
      set_error(std::string("kvx_fit_ridge: device status ") + kvx_status_string(static_cast<kvx_status>(dstat)));
      result = static_cast<kvx_status>(dstat);
    }
  } while (false);
  if (own) cudaFreeAsync(own, st);
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess && result == KVX_OK) {
    set_error(std::string("kvx_fit_ridge: free: ") + cudaGetErrorString(e));
    result = KVX_ERR_CUDA;
  }
  if (result == KVX_OK) timer.finish();
  return result;
}

}  // extern "C"
