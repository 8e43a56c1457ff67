// SIMT kernel: the mapper of Eq. ridge_kv with the Sec. 3.3 RoPE composition, in fp32
// FMA on the CUDA cores.  It runs every configuration the ABI accepts (fp32 or bf16
// caches and weights, head_dim <= 256, per-head or cross-head features, both RoPE
// pair layouts, contiguous or paged targets).  The tensor-core kernel in kvx_tc.cu
// covers the bf16 / head_dim 128 / per-head case at full speed.
//
// One CTA maps TT tokens of one sequence for one (target layer l, K|V, head h):
//   1. gather the k selected source rows (all heads for cross-head), strip the source
//      RoPE from keys in fp32 and round the stripped keys to the cache dtype (the
//      bf16 forward's operand rounding), into shared memory X[TT][F];
//   2. y[c] = sum_f X[f] W[f][c] + b[c] with one thread per output channel c
//      (coalesced reads of the row-major W[F][d]);
//   3. keys: rotate by the target RoPE at the same position; store in the cache dtype.
#include <cuda_bf16.h>

#include "kvx_internal.h"
#include "kvx_rope.cuh"

namespace kvx {
namespace {

constexpr int kSimtThreads = 128;
constexpr int kSimtMaxTT = 16;

struct SimtParams {
  MapArgs a;
  const int32_t* sel;
  const void* W;
  const float* bias;
  int32_t* status;
  int32_t Lt, H, d, k, F, cross, interleaved, cache_bf16, weight_bf16, tt, hf;
  RopeTables rope;
};

__device__ __forceinline__ float load_elem(const void* p, int64_t i, int bf16) {
  return bf16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i])
              : static_cast<const float*>(p)[i];
}

__device__ __forceinline__ void store_elem(void* p, int64_t i, float v, int bf16) {
  if (bf16)
    static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
  else
    static_cast<float*>(p)[i] = v;
}

__device__ __forceinline__ void report(int32_t* status, int code) { atomicCAS(status, 0, code); }

// Rounding to the cache dtype (bf16 round-to-nearest-even, or nothing for fp32 caches).
__device__ __forceinline__ float rc(float x, int bf16) {
  return bf16 ? __bfloat162float(__float2bfloat16_rn(x)) : x;
}

// HF numerics: cos and sin of the fp32 angle fp32(t) * fp32(omega), rounded to the cache
// dtype (the library sincosf, which reduces any fp32 argument).
__device__ __forceinline__ void hf_sincos(int t, float w, int bf16, float* s, float* c) {
  float sv, cv;
  sincosf(__fmul_rn(static_cast<float>(t), w), &sv, &cv);
  *s = rc(sv, bf16);
  *c = rc(cv, bf16);
}

__global__ void __launch_bounds__(kSimtThreads) simt_map_kernel(const __grid_constant__ SimtParams P) {
  extern __shared__ float smem[];
  const int TT = P.tt, F = P.F, d = P.d, H = P.H, k = P.k;
  const int half = d / 2;
  float* X = smem;                                       // [TT][F]
  float* Y = X + TT * F;                                 // [TT][d]
  int* tpos = reinterpret_cast<int*>(Y + TT * d);        // [TT], -1 = row not mapped
  const int t0 = blockIdx.x * TT;
  const int b = blockIdx.y;
  const int h = blockIdx.z % H;
  const int kv = (blockIdx.z / H) % 2;
  const int l = blockIdx.z / (2 * H);
  const MapArgs& a = P.a;

  for (int i = threadIdx.x; i < TT; i += blockDim.x) {
    const int t = t0 + i;
    int p = -1;
    if (t < a.T) {
      p = a.pos[static_cast<int64_t>(b) * a.T + t];
      if (p < 0 || p >= (1 << 24)) {
        report(P.status, KVX_ERR_DEVICE_BOUNDS);
        p = -1;
      }
    }
    tpos[i] = p;
  }
  __syncthreads();

  // 1. gather + strip
  const void* src = kv ? a.src_v : a.src_k;
  const int nh = P.cross ? H : 1;
  const int n_items = TT * k * nh * half;
  for (int it = threadIdx.x; it < n_items; it += blockDim.x) {
    const int i = it % half;
    int r = it / half;
    const int hi = r % nh;
    r /= nh;
    const int j = r % k;
    const int tt = r / k;
    const int p = tpos[tt];
    const int ia = P.interleaved ? 2 * i : i;
    const int ib = P.interleaved ? 2 * i + 1 : i + half;
    float xa = 0.f, xb = 0.f;
    if (p >= 0) {
      const int s = P.sel[l * k + j];
      const int hs = P.cross ? hi : h;
      const int64_t base = s * a.ss[0] + b * a.ss[1] + hs * a.ss[2] + static_cast<int64_t>(t0 + tt) * a.ss[3];
      xa = load_elem(src, base + ia, P.cache_bf16);
      xb = load_elem(src, base + ib, P.cache_bf16);
      if (kv == 0 && P.hf) {
        // the HF rotation with -sin: every product and sum rounded to the cache dtype
        float sn, cs;
        hf_sincos(p, P.rope.ws_hi[i], P.cache_bf16, &sn, &cs);
        const float na = rc(__fadd_rn(rc(__fmul_rn(xa, cs), P.cache_bf16), rc(__fmul_rn(xb, sn), P.cache_bf16)),
                            P.cache_bf16);
        const float nb = rc(__fsub_rn(rc(__fmul_rn(xb, cs), P.cache_bf16), rc(__fmul_rn(xa, sn), P.cache_bf16)),
                            P.cache_bf16);
        xa = na;
        xb = nb;
      } else if (kv == 0) {
        float sn, cs;
        rope_sincos(p, P.rope.ws_hi[i], P.rope.ws_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo,
                    P.rope.inv_two_pi, &sn, &cs);
        // rotation by -t*omega (the strip R_s(t)^-1)
        float na = __fmaf_rn(xa, cs, __fmul_rn(xb, sn));
        float nb = __fmaf_rn(xb, cs, -__fmul_rn(xa, sn));
        if (P.cache_bf16) {
          na = __bfloat162float(__float2bfloat16_rn(na));
          nb = __bfloat162float(__float2bfloat16_rn(nb));
        }
        xa = na;
        xb = nb;
      }
    }
    const int f0 = (j * nh + hi) * d;
    X[tt * F + f0 + ia] = xa;
    X[tt * F + f0 + ib] = xb;
  }
  __syncthreads();

  // 2. contraction y = X W + b
  const size_t wbase = ((static_cast<size_t>(l) * 2 + kv) * H + h) * static_cast<size_t>(F) * d;
  const float* bias = P.bias + ((static_cast<size_t>(l) * 2 + kv) * H + h) * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float acc[kSimtMaxTT];
#pragma unroll
    for (int tt = 0; tt < kSimtMaxTT; ++tt) acc[tt] = 0.f;
    for (int f = 0; f < F; ++f) {
      const float w = load_elem(P.W, wbase + static_cast<size_t>(f) * d + c, P.weight_bf16);
#pragma unroll
      for (int tt = 0; tt < kSimtMaxTT; ++tt)
        if (tt < TT) acc[tt] = __fmaf_rn(X[tt * F + f], w, acc[tt]);
    }
    const float bc = bias[c];
#pragma unroll
    for (int tt = 0; tt < kSimtMaxTT; ++tt)
      if (tt < TT) Y[tt * d + c] = __fadd_rn(acc[tt], bc);
  }
  __syncthreads();

  // 3. target RoPE (keys) and store
  void* dst = kv ? a.tgt_v : a.tgt_k;
  for (int it = threadIdx.x; it < TT * half; it += blockDim.x) {
    const int i = it % half;
    const int tt = it / half;
    const int p = tpos[tt];
    if (p < 0) continue;
    const int ia = P.interleaved ? 2 * i : i;
    const int ib = P.interleaved ? 2 * i + 1 : i + half;
    float ya = Y[tt * d + ia], yb = Y[tt * d + ib];
    if (kv == 0 && P.hf) {
      // the mapped key as a cache-dtype tensor, then the HF rotation at the target angle
      const int bf = P.cache_bf16;
      ya = rc(ya, bf);
      yb = rc(yb, bf);
      float sn, cs;
      hf_sincos(p, P.rope.wt_hi[i], bf, &sn, &cs);
      const float na = rc(__fsub_rn(rc(__fmul_rn(ya, cs), bf), rc(__fmul_rn(yb, sn), bf)), bf);
      const float nb = rc(__fadd_rn(rc(__fmul_rn(yb, cs), bf), rc(__fmul_rn(ya, sn), bf)), bf);
      ya = na;
      yb = nb;
    } else if (kv == 0) {
      float sn, cs;
      rope_sincos(p, P.rope.wt_hi[i], P.rope.wt_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo,
                  P.rope.inv_two_pi, &sn, &cs);
      const float na = __fmaf_rn(ya, cs, -__fmul_rn(yb, sn));
      const float nb = __fmaf_rn(ya, sn, __fmul_rn(yb, cs));
      ya = na;
      yb = nb;
    }
    int64_t base;
    if (!a.paged) {
      base = l * a.ts[0] + b * a.ts[1] + h * a.ts[2] + static_cast<int64_t>(t0 + tt) * a.ts[3];
    } else {
      const int lb = p / a.block_size;
      if (lb >= a.max_blocks) {
        report(P.status, KVX_ERR_DEVICE_BOUNDS);
        continue;
      }
      const int blk = a.block_table[static_cast<int64_t>(b) * a.max_blocks + lb];
      if (blk < 0 || blk >= a.n_blocks) {
        report(P.status, KVX_ERR_DEVICE_BOUNDS);
        continue;
      }
      base = l * a.ts[0] + static_cast<int64_t>(blk) * a.ts[1] + h * a.ts[2] +
             static_cast<int64_t>(p % a.block_size) * a.ts[3];
    }
    store_elem(dst, base + ia, ya, P.cache_bf16);
    store_elem(dst, base + ib, yb, P.cache_bf16);
  }
}

}  // namespace

kvx_status launch_simt(const kvx_ctx* ctx, const MapArgs& a, cudaStream_t stream) {
  SimtParams P{};
  P.a = a;
  P.sel = ctx->d_sel;
  P.W = ctx->d_W;
  P.bias = ctx->d_b;
  P.status = ctx->d_status;
  P.Lt = ctx->Lt;
  P.H = ctx->H;
  P.d = ctx->d;
  P.k = ctx->k;
  P.F = ctx->F;
  P.cross = ctx->head_mix == KVX_CROSS_HEAD;
  P.interleaved = ctx->rope_style == KVX_ROPE_INTERLEAVED;
  P.cache_bf16 = ctx->cache_dtype == KVX_BF16;
  P.weight_bf16 = ctx->weight_dtype == KVX_BF16;
  P.rope = ctx->rope;
  P.hf = ctx->rope_numerics == KVX_ROPE_HF;
  constexpr size_t kSmemBudget = 96 * 1024;
  const size_t per_token = (static_cast<size_t>(ctx->F) + ctx->d) * sizeof(float) + sizeof(int);
  int tt = static_cast<int>(kSmemBudget / per_token);
  tt = tt > kSimtMaxTT ? kSimtMaxTT : tt;
  if (tt < 1) {
    set_error("kvx_map: feature width too large for the SIMT kernel");
    return KVX_ERR_UNSUPPORTED;
  }
  P.tt = tt;
  const size_t smem = per_token * tt;
  cudaError_t e = cudaFuncSetAttribute(simt_map_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: SIMT smem attribute: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  const int64_t zdim = static_cast<int64_t>(ctx->Lt) * 2 * ctx->H;
  if (zdim > 65535 || a.B > 65535) {
    set_error("kvx_map: SIMT grid too large (layers*2*heads or batch > 65535)");
    return KVX_ERR_UNSUPPORTED;
  }
  dim3 grid((a.T + tt - 1) / tt, a.B, static_cast<unsigned>(zdim));
  simt_map_kernel<<<grid, kSimtThreads, smem, stream>>>(P);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: SIMT launch: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

}  // namespace kvx
