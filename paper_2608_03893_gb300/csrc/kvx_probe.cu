// Single-source R^2 probe (Sec. 2.3, Eq. single_source_ols) and the selection scores of
// Sec. 3.2 on the GPU.  For target layer l, source layer l', K|V and head h, the OLS fit
// with intercept of the target head on the source head over N calibration tokens (keys
// RoPE-stripped on both sides) has
//   R^2 = explained / SS_tot,   explained = tr(C^T A^{-1} C),   SS_tot = ||Yc||_F^2,
// with A = Xc^T Xc (128 x 128), C = Xc^T Yc (128 x 128) of the centred columns: the residual
// of the least-squares fit is Yc - Xc A^{-1} C, orthogonal to Xc, so SS_res = SS_tot -
// explained (R^2 pooled over the output channels, variance explained).  With the Cholesky
// factor A = L L^T, explained = ||L^{-1} C||_F^2.  The score is
//   S[l][l'] = (mean_h R^2_K + mean_h R^2_V) / 2.
//
// Steps: the column sums and every block A (one per source layer, K|V, head) and C (one per
// layer pair, K|V, head) on the tensor cores (kvx_gram.cu), SS_tot of each target head from
// the packing pass; then
// 1. probe_factor_kernel: per (K|V, head, source layer) the fp64 Cholesky of A in shared
//    memory and the explicit inverse L^{-1} (forward substitution on the identity), stored
//    transposed in fp32;
// 2. probe_score_kernel: per (K|V, head, source layer) and a group of target layers,
//    Z = L^{-1} C with FFMA 8 x 8 register tiles over the lower triangle, explained = sum
//    Z^2, R^2 in fp64;
// 3. probe_reduce_kernel: head average and the K/V mean.
// Top-k on the device (kvx_select_topk_device): one thread per target layer.
#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <string>
#include <vector>

#include "kvx_gram.h"
#include "kvx_internal.h"

namespace kvx {
namespace {

constexpr int kPD = 128;
constexpr int kPTri = kPD * (kPD + 1) / 2;       // packed lower triangle
constexpr int kPTargets = 16;                     // target layers per score CTA
constexpr int kNotPd = 101;                       // internal status: a source Gram block is singular

__device__ __forceinline__ int tri(int i, int j) { return i * (i + 1) / 2 + j; }   // j <= i

__device__ __forceinline__ void preport(int32_t* status, int code) { atomicCAS(status, 0, code); }

// grid: 2 H L_s systems, 256 threads, dynamic shared memory 2 kPTri doubles (L and L^{-1}).
// A [sys][128][128] fp32 -> linvT [sys][128][128] fp32 with linvT[k][i] = (L^{-1})[i][k].
__global__ void __launch_bounds__(256) probe_factor_kernel(const float* __restrict__ A, float* __restrict__ linvT,
                                                           int32_t* status) {
  extern __shared__ double psh[];
  double* L = psh;                 // packed lower triangle
  double* X = psh + kPTri;         // packed lower triangle of L^{-1}
  const int tid = threadIdx.x;
  const float* a = A + static_cast<size_t>(blockIdx.x) * kPD * kPD;
  for (int e = tid; e < kPTri; e += blockDim.x) {
    int i = static_cast<int>((sqrtf(8.f * e + 1.f) - 1.f) * 0.5f);
    while (tri(i + 1, 0) <= e) ++i;
    while (tri(i, 0) > e) --i;
    const int j = e - tri(i, 0);
    L[e] = static_cast<double>(a[i * kPD + j]);
  }
  __syncthreads();
  __shared__ int bad;
  if (tid == 0) bad = 0;
  __syncthreads();
  // right-looking Cholesky, one column at a time
  for (int j = 0; j < kPD; ++j) {
    if (tid == 0) {
      const double d = L[tri(j, j)];
      if (!(d > 0.0)) bad = 1;
      L[tri(j, j)] = d > 0.0 ? sqrt(d) : 1.0;
    }
    __syncthreads();
    const double djj = L[tri(j, j)];
    for (int i = j + 1 + tid; i < kPD; i += blockDim.x) L[tri(i, j)] /= djj;
    __syncthreads();
    // trailing update of rows i > j, columns j < m <= i
    const int rows = kPD - j - 1;
    const int cnt = rows * (rows + 1) / 2;
    for (int e = tid; e < cnt; e += blockDim.x) {
      int r = static_cast<int>((sqrtf(8.f * e + 1.f) - 1.f) * 0.5f);
      while ((r + 1) * (r + 2) / 2 <= e) ++r;
      while (r * (r + 1) / 2 > e) --r;
      const int c = e - r * (r + 1) / 2;
      const int i = j + 1 + r, m = j + 1 + c;
      L[tri(i, m)] -= L[tri(i, j)] * L[tri(m, j)];
    }
    __syncthreads();
  }
  if (bad) {
    if (tid == 0) preport(status, kNotPd);
    return;
  }
  // L^{-1} by forward substitution on the identity: thread = column c (two threads per
  // column split the inner sums over m)
  const int c = tid & (kPD - 1), half = tid >> 7;
  __shared__ double part[256];
  for (int i = 0; i < kPD; ++i) {
    double s = 0.0;
    if (i >= c)
      for (int m = c + half; m < i; m += 2) s += L[tri(i, m)] * X[tri(m, c)];
    part[tid] = s;
    __syncthreads();
    if (half == 0 && i >= c) X[tri(i, c)] = ((i == c ? 1.0 : 0.0) - part[c] - part[c + kPD]) / L[tri(i, i)];
    __syncthreads();
  }
  float* out = linvT + static_cast<size_t>(blockIdx.x) * kPD * kPD;
  for (int e = tid; e < kPD * kPD; e += blockDim.x) {
    const int k = e / kPD, i = e % kPD;         // out[k][i] = X[i][k]
    out[e] = i >= k ? static_cast<float>(X[tri(i, k)]) : 0.f;
  }
}

// grid: (2 H L_s, ceil(L_t / 16)), 256 threads, 128 KB dynamic shared memory.
// For each target layer t of the group: Z = L^{-1} C_ts, r2[kv][h][t][s] = sum Z^2 / SS_tot.
__global__ void __launch_bounds__(256) probe_score_kernel(const float* __restrict__ linvT, const float* __restrict__ C,
                                                          const double* __restrict__ sumsq, double* __restrict__ r2,
                                                          int H, int Ls, int Lt, int tslot0) {
  extern __shared__ __align__(16) float fsh[];
  float* lt = fsh;                  // [k][i]
  float* cb = fsh + kPD * kPD;      // [k][j]
  __shared__ float red[8];
  const int sys = blockIdx.x;       // (kv * H + h) * Ls + s
  const int s = sys % Ls, kvh = sys / Ls;
  const int h = kvh % H, kv = kvh / H;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  {
    const float4* src = reinterpret_cast<const float4*>(linvT + static_cast<size_t>(sys) * kPD * kPD);
    for (int e = tid; e < kPD * kPD / 4; e += blockDim.x) reinterpret_cast<float4*>(lt)[e] = src[e];
  }
  const int t_end = min(Lt, (blockIdx.y + 1) * kPTargets);
  for (int t = blockIdx.y * kPTargets; t < t_end; ++t) {
    __syncthreads();   // the previous target's reads of cb are done
    const float4* src =
        reinterpret_cast<const float4*>(C + ((static_cast<size_t>(kvh) * Ls + s) * Lt + t) * kPD * kPD);
    for (int e = tid; e < kPD * kPD / 4; e += blockDim.x) reinterpret_cast<float4*>(cb)[e] = src[e];
    __syncthreads();
    float acc[8][8];
#pragma unroll
    for (int x = 0; x < 8; ++x)
#pragma unroll
      for (int y = 0; y < 8; ++y) acc[x][y] = 0.f;
    const int k_end = 8 * ty + 8;   // L^{-1} rows 8ty.. are zero past column 8ty+7
#pragma unroll 4
    for (int k = 0; k < k_end; ++k) {
      const float4 a0 = *reinterpret_cast<const float4*>(&lt[k * kPD + 8 * ty]);
      const float4 a1 = *reinterpret_cast<const float4*>(&lt[k * kPD + 8 * ty + 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&cb[k * kPD + 8 * tx]);
      const float4 b1 = *reinterpret_cast<const float4*>(&cb[k * kPD + 8 * tx + 4]);
      const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int x = 0; x < 8; ++x)
#pragma unroll
        for (int y = 0; y < 8; ++y) acc[x][y] = __fmaf_rn(av[x], bv[y], acc[x][y]);
    }
    float sq = 0.f;
#pragma unroll
    for (int x = 0; x < 8; ++x)
#pragma unroll
      for (int y = 0; y < 8; ++y) sq = __fmaf_rn(acc[x][y], acc[x][y], sq);
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, d);
    if ((tid & 31) == 0) red[tid >> 5] = sq;
    __syncthreads();
    if (tid == 0) {
      double e = 0.0;
      for (int w = 0; w < 8; ++w) e += static_cast<double>(red[w]);
      const double tot = sumsq[(static_cast<size_t>(tslot0 + t) * 2 + kv) * H + h];
      r2[((static_cast<size_t>(kv) * H + h) * Lt + t) * Ls + s] = tot > 0.0 ? e / tot : 0.0;
    }
  }
}

// scores[t][s] = (mean_h r2[0][h][t][s] + mean_h r2[1][h][t][s]) / 2; r2_kv (optional)
// [2][t][s] the head averages.
__global__ void probe_reduce_kernel(const double* __restrict__ r2, double* __restrict__ scores,
                                    double* __restrict__ r2_kv, int H, int Ls, int Lt) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= Lt * Ls) return;
  double m[2] = {0.0, 0.0};
  for (int kv = 0; kv < 2; ++kv) {
    for (int h = 0; h < H; ++h) m[kv] += r2[(static_cast<size_t>(kv) * H + h) * Lt * Ls + i];
    m[kv] /= H;
    if (r2_kv) r2_kv[static_cast<size_t>(kv) * Lt * Ls + i] = m[kv];
  }
  scores[i] = 0.5 * (m[0] + m[1]);
}

// One thread per target layer: the k largest scores, ties to the lower source index, the
// row returned in ascending source order (as kvx_select_topk).  A NaN score raises status.
__global__ void topk_kernel(const double* __restrict__ scores, int Lt, int Ls, int k, int32_t* __restrict__ out,
                            int32_t* status) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= Lt) return;
  const double* row = scores + static_cast<size_t>(t) * Ls;
  int32_t* o = out + static_cast<size_t>(t) * k;
  for (int s = 0; s < Ls; ++s)
    if (isnan(row[s])) {
      preport(status, KVX_ERR_INVALID_ARG);
      for (int j = 0; j < k; ++j) o[j] = j;
      return;
    }
  // select k times the best not yet taken: higher score, then lower index
  for (int j = 0; j < k; ++j) {
    int best = -1;
    for (int s = 0; s < Ls; ++s) {
      bool taken = false;
      for (int q = 0; q < j; ++q) taken |= o[q] == s;
      if (taken) continue;
      if (best < 0 || row[s] > row[best]) best = s;
    }
    o[j] = best;
  }
  for (int a = 1; a < k; ++a) {   // ascending source order
    const int32_t v = o[a];
    int b = a - 1;
    while (b >= 0 && o[b] > v) {
      o[b + 1] = o[b];
      --b;
    }
    o[b + 1] = v;
  }
}

kvx_status pfail(const std::string& m, kvx_status s) {
  set_error(m);
  return s;
}

const char* check_probe_config(const kvx_probe_config* cfg) {
  if (!cfg) return "NULL argument";
  if (cfg->head_dim != kPD) return "head_dim must be 128";
  if (cfg->src_layers < 1 || cfg->tgt_layers < 1 || cfg->n_kv_heads < 1) return "layer / head counts out of range";
  if (!(cfg->src_rope_theta > 1.0) || !(cfg->tgt_rope_theta > 1.0) || !std::isfinite(cfg->src_rope_theta) ||
      !std::isfinite(cfg->tgt_rope_theta))
    return "the RoPE bases must be finite and > 1";
  if (cfg->workspace_bytes != 0 && !cfg->workspace) return "workspace_bytes without a workspace";
  if (cfg->rope_numerics != KVX_ROPE_EXACT && cfg->rope_numerics != KVX_ROPE_HF) return "bad rope_numerics";
  if (const char* why = check_rope_scaling(cfg->src_rope_scaling)) return why;
  if (const char* why = check_rope_scaling(cfg->tgt_rope_scaling)) return why;
  if (reinterpret_cast<uintptr_t>(cfg->workspace) & 255u) return "workspace must be 256-byte aligned";
  return nullptr;
}

// Sizes of the probe's own device pieces and its operand slots (every layer of both models).
struct ProbePlan {
  size_t blk = static_cast<size_t>(kPD) * kPD, n_src = 0, n_cross = 0, sums_n = 0, sumsq_n = 0, r2_n = 0;
  size_t own_bytes = 0, n_blocks = 0;
};

ProbePlan plan_probe(const kvx_probe_config* cfg, GramSpec* G) {
  ProbePlan p;
  const int Ls = cfg->src_layers, Lt = cfg->tgt_layers, H = cfg->n_kv_heads;
  G->slot_side.clear();
  G->slot_layer.clear();
  for (int L = 0; L < Ls; ++L) {
    G->slot_side.push_back(0);
    G->slot_layer.push_back(L);
  }
  for (int l = 0; l < Lt; ++l) {
    G->slot_side.push_back(1);
    G->slot_layer.push_back(l);
  }
  G->H = H;
  p.n_src = static_cast<size_t>(2) * H * Ls;
  p.n_cross = p.n_src * Lt;
  p.sums_n = static_cast<size_t>(2) * (Ls + Lt) * H * kPD;
  p.sumsq_n = static_cast<size_t>(Ls + Lt) * 2 * H;
  p.r2_n = static_cast<size_t>(2) * H * Lt * Ls;
  auto al = [](size_t n) { return (n + 255) / 256 * 256; };
  p.own_bytes = al((p.sums_n + p.sumsq_n) * 8) + al(p.r2_n * 8) + al(p.n_src * p.blk * 4) * 2 +
                al(p.n_cross * p.blk * 4) + al(4);
  p.n_blocks = p.n_src * (Lt + 1);
  return p;
}

}  // namespace
}  // namespace kvx

extern "C" {

KVX_API int64_t kvx_r2_probe_workspace_bytes(const kvx_probe_config* cfg, int32_t batch, int32_t tokens_per_seq) {
  using namespace kvx;
  if (check_probe_config(cfg) || batch < 1 || tokens_per_seq < 1) return -1;
  GramSpec G;
  const ProbePlan p = plan_probe(cfg, &G);
  const int64_t N = static_cast<int64_t>(batch) * tokens_per_seq;
  const size_t np = static_cast<size_t>((N + 63) / 64 * 64);
  return static_cast<int64_t>(p.own_bytes + gram_fixed_bytes(G, p.n_blocks) + gram_bytes_per_token(G) * np + 1024);
}

KVX_API kvx_status kvx_r2_probe(const kvx_probe_config* cfg, const kvx_src* src, const kvx_src* tgt, int32_t batch,
                                int32_t tokens_per_seq, const int32_t* positions, double* scores, double* r2_kv,
                                void* stream) {
  using namespace kvx;
  NvtxRange range("kvx_r2_probe");
  set_error("");
  auto bad = [](const char* m) { return pfail(std::string("kvx_r2_probe: ") + m, KVX_ERR_INVALID_ARG); };
  if (const char* why = check_probe_config(cfg)) return bad(why);
  if (!src || !tgt || !positions || !scores) return bad("NULL argument");
  if (batch < 1 || tokens_per_seq < 1) return bad("batch and tokens_per_seq must be >= 1");
  if (static_cast<int64_t>(batch) * tokens_per_seq <= kPD)
    return bad("need more than 128 calibration tokens (the source Gram blocks are singular otherwise)");
  const kvx_src* cs[2] = {src, tgt};
  for (const kvx_src* c : cs) {
    if (!c->k || !c->v) return bad("NULL cache pointer");
    if ((reinterpret_cast<uintptr_t>(c->k) | reinterpret_cast<uintptr_t>(c->v)) & 15u)
      return bad("cache pointers must be 16-byte aligned");
    for (int i = 0; i < 4; ++i)
      if (c->stride[i] < 0 || c->stride[i] % 8 != 0) return bad("strides must be non-negative multiples of 8");
    if (c->stride[3] < kPD) return bad("token stride smaller than head_dim");
  }
  if (reinterpret_cast<uintptr_t>(positions) & 3u) return bad("positions must be 4-byte aligned");
  if ((reinterpret_cast<uintptr_t>(scores) | reinterpret_cast<uintptr_t>(r2_kv)) & 7u)
    return bad("scores and r2_kv must be 8-byte aligned");

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  int dev = 0, sms = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return pfail(std::string("kvx_r2_probe: device query: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
  kvx_ctx tmp;   // for the RoPE tables only
  tmp.d = kPD;
  tmp.theta_s = cfg->src_rope_theta;
  tmp.theta_t = cfg->tgt_rope_theta;
  set_rope_scaling(&tmp, cfg->src_rope_scaling, cfg->tgt_rope_scaling);
  fill_rope(&tmp);

  const int Ls = cfg->src_layers, Lt = cfg->tgt_layers, H = cfg->n_kv_heads;
  GramSpec G;
  const ProbePlan pl = plan_probe(cfg, &G);
  G.cache[0] = GramCache{src->k, src->v, {src->stride[0], src->stride[1], src->stride[2], src->stride[3]}};
  G.cache[1] = GramCache{tgt->k, tgt->v, {tgt->stride[0], tgt->stride[1], tgt->stride[2], tgt->stride[3]}};
  G.pos = positions;
  G.B = batch;
  G.T = tokens_per_seq;
  G.Ls = Ls;
  G.Lt = Lt;
  G.rope = tmp.rope;
  G.hf = cfg->rope_numerics == KVX_ROPE_HF;
  G.sm_count = sms;
  const size_t blk = pl.blk;
  const bool caller_ws = cfg->workspace != nullptr;
  Scratch S;
  char* own = nullptr;
  if (caller_ws) {
    S.p = static_cast<char*>(cfg->workspace);
    S.bytes = static_cast<size_t>(cfg->workspace_bytes);
    if (S.bytes < pl.own_bytes + gram_fixed_bytes(G, pl.n_blocks))
      return bad("workspace too small (see kvx_r2_probe_workspace_bytes)");
  } else {
    if ((e = cudaMallocAsync(reinterpret_cast<void**>(&own), pl.own_bytes, st)) != cudaSuccess)
      return pfail(std::string("kvx_r2_probe: workspace: ") + cudaGetErrorString(e), KVX_ERR_OOM);
    S.p = own;
    S.bytes = pl.own_bytes;
  }
  double* sums = reinterpret_cast<double*>(S.take((pl.sums_n + pl.sumsq_n) * 8));
  double* sumsq = sums + pl.sums_n;
  double* r2 = reinterpret_cast<double*>(S.take(pl.r2_n * 8));
  float* A = reinterpret_cast<float*>(S.take(pl.n_src * blk * 4));
  float* linvT = reinterpret_cast<float*>(S.take(pl.n_src * blk * 4));
  float* C = reinterpret_cast<float*>(S.take(pl.n_cross * blk * 4));
  int32_t* status = reinterpret_cast<int32_t*>(S.take(4));
  if (!caller_ws) S = Scratch{};
  G.sums = sums;
  G.sumsq = sumsq;
  G.status = status;
  kvx_status result = KVX_OK;
  PhaseTimer timer(st);
  do {
    if ((e = cudaMemsetAsync(sums, 0, (pl.sums_n + pl.sumsq_n) * 8, st)) != cudaSuccess ||
        (e = cudaMemsetAsync(status, 0, 4, st)) != cudaSuccess) {
      result = pfail(std::string("kvx_r2_probe: setup: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
      break;
    }
    std::vector<GramBlock> blocks;
    blocks.reserve(pl.n_blocks);
    for (int kv = 0; kv < 2; ++kv)
      for (int h = 0; h < H; ++h)
        for (int s = 0; s < Ls; ++s) {
          const size_t sys = (static_cast<size_t>(kv) * H + h) * Ls + s;
          blocks.push_back(GramBlock{s, s, kv, h, A + sys * blk});
          for (int t = 0; t < Lt; ++t) blocks.push_back(GramBlock{s, Ls + t, kv, h, C + (sys * Lt + t) * blk});
        }
    size_t budget = 0;
    if (!caller_ws) {
      size_t free_b = 0, total_b = 0;
      if ((e = cudaMemGetInfo(&free_b, &total_b)) != cudaSuccess) {
        result = pfail(std::string("kvx_r2_probe: memory query: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
        break;
      }
      budget = std::min<size_t>(free_b / 2, static_cast<size_t>(32) << 30);
    }
    Scratch* sp = caller_ws ? &S : nullptr;
    if ((result = gram_sums(G, st, &timer, sp)) != KVX_OK ||
        (result = gram_blocks(G, blocks, budget, st, &timer, sp)) != KVX_OK) {
      set_error(std::string("kvx_r2_probe: ") + kvx_last_error());
      break;
    }
    const size_t fsmem = static_cast<size_t>(2) * kPTri * 8;
    const size_t ssmem = static_cast<size_t>(2) * blk * 4;
    if ((e = cudaFuncSetAttribute(probe_factor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(fsmem))) != cudaSuccess ||
        (e = cudaFuncSetAttribute(probe_score_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(ssmem))) != cudaSuccess) {
      result = pfail(std::string("kvx_r2_probe: smem attribute: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
      break;
    }
    timer.begin(3);
    probe_factor_kernel<<<static_cast<unsigned>(pl.n_src), 256, fsmem, st>>>(A, linvT, status);
    probe_score_kernel<<<dim3(static_cast<unsigned>(pl.n_src), static_cast<unsigned>((Lt + kPTargets - 1) / kPTargets)),
                         256, ssmem, st>>>(linvT, C, sumsq, r2, H, Ls, Lt, Ls);
    probe_reduce_kernel<<<static_cast<unsigned>((static_cast<int64_t>(Lt) * Ls + 255) / 256), 256, 0, st>>>(
        r2, scores, r2_kv, H, Ls, Lt);
    timer.end();
    if ((e = cudaGetLastError()) != cudaSuccess) {
      result = pfail(std::string("kvx_r2_probe: launch: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
      break;
    }
    int32_t dstat = 0;
    if ((e = cudaMemcpyAsync(&dstat, status, 4, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
        (e = cudaStreamSynchronize(st)) != cudaSuccess) {
      result = pfail(std::string("kvx_r2_probe: run: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
      break;
    }
    if (dstat == kNotPd) {
      result = pfail("kvx_r2_probe: a source Gram block is singular (a constant channel, or too few distinct tokens)",
                     KVX_ERR_INVALID_ARG);
    } else if (dstat == KVX_ERR_DEVICE_BOUNDS) {
      result = pfail("kvx_r2_probe: a position is outside [0, 2^24)", KVX_ERR_DEVICE_BOUNDS);
    } else if (dstat != 0) {
      result = pfail(std::string("kvx_r2_probe: device status ") + kvx_status_string(static_cast<kvx_status>(dstat)),
                     static_cast<kvx_status>(dstat));
    }
  } while (false);
  if (own) cudaFreeAsync(own, st);
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess && result == KVX_OK)
    result = pfail(std::string("kvx_r2_probe: free: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
  if (result == KVX_OK) timer.finish();
  return result;
}

KVX_API kvx_status kvx_select_topk_device(const double* scores, int32_t tgt_layers, int32_t src_layers, int32_t k,
                                          int32_t* out, void* stream) {
  using namespace kvx;
  set_error("");
  if (!scores || !out) return pfail("kvx_select_topk_device: NULL pointer", KVX_ERR_INVALID_ARG);
  if (tgt_layers <= 0 || src_layers <= 0)
    return pfail("kvx_select_topk_device: layer counts must be positive", KVX_ERR_INVALID_ARG);
  if (k < 1 || k > src_layers) return pfail("kvx_select_topk_device: k must be in [1, src_layers]", KVX_ERR_INVALID_ARG);
  if ((reinterpret_cast<uintptr_t>(scores) & 7u) || (reinterpret_cast<uintptr_t>(out) & 3u))
    return pfail("kvx_select_topk_device: misaligned pointer", KVX_ERR_INVALID_ARG);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  int32_t* status = nullptr;
  if ((e = cudaMallocAsync(reinterpret_cast<void**>(&status), 4, st)) != cudaSuccess)
    return pfail(std::string("kvx_select_topk_device: ") + cudaGetErrorString(e), KVX_ERR_OOM);
  kvx_status result = KVX_OK;
  int32_t dstat = 0;
  if ((e = cudaMemsetAsync(status, 0, 4, st)) == cudaSuccess) {
    topk_kernel<<<(tgt_layers + 127) / 128, 128, 0, st>>>(scores, tgt_layers, src_layers, k, out, status);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(&dstat, status, 4, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFreeAsync(status, st);
  if (e != cudaSuccess) {
    result = pfail(std::string("kvx_select_topk_device: ") + cudaGetErrorString(e), KVX_ERR_CUDA);
  } else if (dstat != 0) {
    result = pfail("kvx_select_topk_device: NaN score", KVX_ERR_INVALID_ARG);
  }
  return result;
}

}  // extern "C"
