// Host side of libkvx: argument validation, top-k selection, device copies of the
// mapper, kernel dispatch and the device status word.  See include/kvx.h for the ABI.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <numeric>
#include <string>
#include <vector>

#include "kvx_internal.h"
#include "kvx_xh.h"

namespace kvx {

static thread_local std::string g_last_error;

void set_error(const std::string& msg) { g_last_error = msg; }

static kvx_status fail(kvx_status s, const std::string& msg) {
  set_error(msg);
  return s;
}

static kvx_status cuda_fail(cudaError_t e, const char* what) {
  return fail(KVX_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

// Restores the caller's current device on scope exit.
struct DeviceGuard {
  int prev = -1;
  cudaError_t err = cudaSuccess;
  explicit DeviceGuard(int dev) {
    err = cudaGetDevice(&prev);
    if (err == cudaSuccess && prev != dev) err = cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

// Top-k per row: order by (score descending, index ascending), keep k, sort ascending.
static void topk_rows(const double* scores, int lt, int ls, int k, int32_t* out) {
  std::vector<int32_t> idx(ls);
  for (int l = 0; l < lt; ++l) {
    const double* row = scores + static_cast<size_t>(l) * ls;
    std::iota(idx.begin(), idx.end(), 0);
    std::stable_sort(idx.begin(), idx.end(), [row](int32_t a, int32_t b) {
      if (row[a] != row[b]) return row[a] > row[b];
      return a < b;
    });
    std::sort(idx.begin(), idx.begin() + k);
    std::copy(idx.begin(), idx.begin() + k, out + static_cast<size_t>(l) * k);
  }
}

static float bf16_to_float(uint16_t v) {
  uint32_t u = static_cast<uint32_t>(v) << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

const char* check_rope_scaling(const kvx_rope_scaling* s) {
  if (!s) return nullptr;
  if (!(s->factor >= 1.0) || !std::isfinite(s->factor)) return "rope scaling factor must be finite and >= 1";
  if (!(s->low_freq_factor > 0.0) || !(s->high_freq_factor > s->low_freq_factor) ||
      !std::isfinite(s->high_freq_factor))
    return "rope scaling needs 0 < low_freq_factor < high_freq_factor";
  if (!(s->original_max_position > 0.0) || !std::isfinite(s->original_max_position))
    return "rope scaling original_max_position must be > 0";
  return nullptr;
}

void set_rope_scaling(kvx_ctx* c, const kvx_rope_scaling* src, const kvx_rope_scaling* tgt) {
  c->scale_s_on = src != nullptr;
  c->scale_t_on = tgt != nullptr;
  if (src) c->scale_s = *src;
  if (tgt) c->scale_t = *tgt;
}

// Llama-3 scaling of one inverse frequency (kvx_rope_scaling in kvx.h), in double.
static double scaled_omega(double w, const kvx_rope_scaling& s) {
  const double two_pi = 6.283185307179586476925286766559;
  const double wavelen = two_pi / w;
  const double lo_wavelen = s.original_max_position / s.low_freq_factor;
  const double hi_wavelen = s.original_max_position / s.high_freq_factor;
  if (wavelen < hi_wavelen) return w;
  if (wavelen > lo_wavelen) return w / s.factor;
  const double sm = (s.original_max_position / wavelen - s.low_freq_factor) / (s.high_freq_factor - s.low_freq_factor);
  return (1.0 - sm) * w / s.factor + sm * w;
}

void fill_rope(kvx_ctx* c) {
  const int half = c->d / 2;
  for (int i = 0; i < half; ++i) {
    const double e = -2.0 * i / c->d;
    double ws = std::pow(c->theta_s, e), wt = std::pow(c->theta_t, e);
    if (c->scale_s_on) ws = scaled_omega(ws, c->scale_s);
    if (c->scale_t_on) wt = scaled_omega(wt, c->scale_t);
    c->rope.ws_hi[i] = static_cast<float>(ws);
    c->rope.ws_lo[i] = static_cast<float>(ws - static_cast<double>(c->rope.ws_hi[i]));
    c->rope.wt_hi[i] = static_cast<float>(wt);
    c->rope.wt_lo[i] = static_cast<float>(wt - static_cast<double>(c->rope.wt_hi[i]));
  }
  const double two_pi = 6.283185307179586476925286766559;
  c->rope.two_pi_hi = static_cast<float>(two_pi);
  c->rope.two_pi_lo = static_cast<float>(two_pi - static_cast<double>(c->rope.two_pi_hi));
  c->rope.inv_two_pi = static_cast<float>(1.0 / two_pi);
}

static void free_ctx(kvx_ctx* c) {
  if (!c) return;
  cudaFree(c->d_sel);
  cudaFree(c->d_W);
  cudaFree(c->d_b);
  cudaFree(c->d_Wt);
  cudaFree(c->d_plan);
  cudaFree(c->d_status);
  cudaFree(c->d_ws);
  delete c;
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace kvx

using namespace kvx;

extern "C" {

const char* kvx_last_error(void) { return g_last_error.c_str(); }

const char* kvx_status_string(kvx_status s) {
  switch (s) {
    case KVX_OK: return "KVX_OK";
    case KVX_ERR_INVALID_ARG: return "KVX_ERR_INVALID_ARG: invalid argument";
    case KVX_ERR_UNSUPPORTED: return "KVX_ERR_UNSUPPORTED: unsupported configuration";
    case KVX_ERR_OOM: return "KVX_ERR_OOM: device allocation failed";
    case KVX_ERR_CUDA: return "KVX_ERR_CUDA: CUDA error";
    case KVX_ERR_TIMEOUT: return "KVX_ERR_TIMEOUT: a device wait ran out";
    case KVX_ERR_DEVICE_BOUNDS: return "KVX_ERR_DEVICE_BOUNDS: position or block index out of range";
  }
  return "unknown kvx_status";
}

int64_t kvx_mapper_params(int32_t tgt_layers, int32_t n_kv_heads, int32_t head_dim, int32_t k,
                          int32_t head_mix) {
  if (tgt_layers <= 0 || n_kv_heads <= 0 || head_dim <= 0 || k <= 0) return -1;
  int64_t feat = static_cast<int64_t>(k) * head_dim;
  if (head_mix == KVX_CROSS_HEAD) feat *= n_kv_heads;
  else if (head_mix != KVX_PER_HEAD) return -1;
  return 2 * static_cast<int64_t>(tgt_layers) * n_kv_heads * feat * head_dim;
}

kvx_status kvx_select_topk(const double* scores, int32_t tgt_layers, int32_t src_layers, int32_t k,
                           int32_t* out) {
  g_last_error.clear();
  if (!scores || !out) return fail(KVX_ERR_INVALID_ARG, "kvx_select_topk: NULL pointer");
  if (tgt_layers <= 0 || src_layers <= 0)
    return fail(KVX_ERR_INVALID_ARG, "kvx_select_topk: layer counts must be positive");
  if (k < 1 || k > src_layers)
    return fail(KVX_ERR_INVALID_ARG, "kvx_select_topk: k must be in [1, src_layers]");
  for (int64_t i = 0; i < static_cast<int64_t>(tgt_layers) * src_layers; ++i)
    if (std::isnan(scores[i])) return fail(KVX_ERR_INVALID_ARG, "kvx_select_topk: NaN score");
  topk_rows(scores, tgt_layers, src_layers, k, out);
  return KVX_OK;
}

kvx_status kvx_create(const kvx_config* cfg, int device, kvx_ctx** out) {
  g_last_error.clear();
  if (!out) return fail(KVX_ERR_INVALID_ARG, "kvx_create: out is NULL");
  *out = nullptr;
  if (!cfg) return fail(KVX_ERR_INVALID_ARG, "kvx_create: cfg is NULL");
  const kvx_config& c = *cfg;
  if (c.src_layers <= 0 || c.tgt_layers <= 0 || c.n_kv_heads <= 0 || c.head_dim <= 0)
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: layer, head and head_dim counts must be positive");
  if (c.head_dim % 2 != 0) return fail(KVX_ERR_UNSUPPORTED, "kvx_create: head_dim must be even");
  if (c.head_dim > kMaxHeadDim) return fail(KVX_ERR_UNSUPPORTED, "kvx_create: head_dim > 256");
  if (c.k < 1 || c.k > c.src_layers)
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: k must be in [1, src_layers]");
  if (c.rope_style != KVX_ROPE_HALF && c.rope_style != KVX_ROPE_INTERLEAVED)
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: bad rope_style");
  if ((c.cache_dtype != KVX_F32 && c.cache_dtype != KVX_BF16) ||
      (c.weight_dtype != KVX_F32 && c.weight_dtype != KVX_BF16))
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: bad dtype");
  if (c.head_mix != KVX_PER_HEAD && c.head_mix != KVX_CROSS_HEAD)
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: bad head_mix");
  if (c.reserved != 0) return fail(KVX_ERR_INVALID_ARG, "kvx_create: reserved must be 0");
  if (c.rope_numerics != KVX_ROPE_EXACT && c.rope_numerics != KVX_ROPE_HF)
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: bad rope_numerics");
  if (const char* why = check_rope_scaling(c.src_rope_scaling))
    return fail(KVX_ERR_INVALID_ARG, std::string("kvx_create: source ") + why);
  if (const char* why = check_rope_scaling(c.tgt_rope_scaling))
    return fail(KVX_ERR_INVALID_ARG, std::string("kvx_create: target ") + why);
  if (!(c.src_rope_theta > 1.0) || !(c.tgt_rope_theta > 1.0) || !std::isfinite(c.src_rope_theta) ||
      !std::isfinite(c.tgt_rope_theta))
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: rope thetas must be finite and > 1");
  if (!c.W) return fail(KVX_ERR_INVALID_ARG, "kvx_create: W is NULL");
  if (!c.selection && !c.selection_scores)
    return fail(KVX_ERR_INVALID_ARG, "kvx_create: need a selection or selection_scores");

  auto* ctx = new kvx_ctx();
  ctx->device = device;
  ctx->Ls = c.src_layers;
  ctx->Lt = c.tgt_layers;
  ctx->H = c.n_kv_heads;
  ctx->d = c.head_dim;
  ctx->k = c.k;
  ctx->head_mix = c.head_mix;
  ctx->F = c.k * c.head_dim * (c.head_mix == KVX_CROSS_HEAD ? c.n_kv_heads : 1);
  ctx->rope_style = c.rope_style;
  ctx->cache_dtype = c.cache_dtype;
  ctx->weight_dtype = c.weight_dtype;
  ctx->theta_s = c.src_rope_theta;
  ctx->theta_t = c.tgt_rope_theta;

  // selection table
  ctx->sel.resize(static_cast<size_t>(ctx->Lt) * ctx->k);
  if (c.selection) {
    std::copy(c.selection, c.selection + ctx->sel.size(), ctx->sel.begin());
    for (int l = 0; l < ctx->Lt; ++l) {
      std::vector<int32_t> row(ctx->sel.begin() + l * ctx->k, ctx->sel.begin() + (l + 1) * ctx->k);
      for (int32_t s : row)
        if (s < 0 || s >= ctx->Ls) {
          free_ctx(ctx);
          return fail(KVX_ERR_INVALID_ARG, "kvx_create: selection entry outside [0, src_layers)");
        }
      std::sort(row.begin(), row.end());
      if (std::adjacent_find(row.begin(), row.end()) != row.end()) {
        free_ctx(ctx);
        return fail(KVX_ERR_INVALID_ARG, "kvx_create: duplicate source layer in a selection row");
      }
    }
  } else {
    kvx_status s = kvx_select_topk(c.selection_scores, ctx->Lt, ctx->Ls, ctx->k, ctx->sel.data());
    if (s != KVX_OK) {
      free_ctx(ctx);
      return s;
    }
  }
  set_rope_scaling(ctx, c.src_rope_scaling, c.tgt_rope_scaling);
  ctx->rope_numerics = c.rope_numerics;
  fill_rope(ctx);

  DeviceGuard guard(device);
  if (guard.err != cudaSuccess) {
    free_ctx(ctx);
    return cuda_fail(guard.err, "kvx_create: cudaSetDevice");
  }
  cudaError_t e = cudaDeviceGetAttribute(&ctx->sm_count, cudaDevAttrMultiProcessorCount, device);
  if (e != cudaSuccess) {
    free_ctx(ctx);
    return cuda_fail(e, "kvx_create: device query");
  }

  const size_t n_w = static_cast<size_t>(ctx->Lt) * 2 * ctx->H * ctx->F * ctx->d;
  const size_t w_bytes = n_w * (ctx->weight_dtype == KVX_BF16 ? 2 : 4);
  const size_t n_b = static_cast<size_t>(ctx->Lt) * 2 * ctx->H * ctx->d;
  std::vector<float> bias(n_b, 0.0f);
  if (c.b) {
    if (ctx->weight_dtype == KVX_BF16) {
      const uint16_t* bb = static_cast<const uint16_t*>(c.b);
      for (size_t i = 0; i < n_b; ++i) bias[i] = bf16_to_float(bb[i]);
    } else {
      std::memcpy(bias.data(), c.b, n_b * 4);
    }
  }
  if ((e = cudaMalloc(&ctx->d_sel, ctx->sel.size() * 4)) != cudaSuccess ||
      (e = cudaMalloc(&ctx->d_W, w_bytes)) != cudaSuccess ||
      (e = cudaMalloc(&ctx->d_b, n_b * 4)) != cudaSuccess ||
      (e = cudaMalloc(&ctx->d_status, 4)) != cudaSuccess) {
    free_ctx(ctx);
    return fail(KVX_ERR_OOM, std::string("kvx_create: cudaMalloc: ") + cudaGetErrorString(e));
  }
  if ((e = cudaMemcpy(ctx->d_sel, ctx->sel.data(), ctx->sel.size() * 4, cudaMemcpyHostToDevice)) !=
          cudaSuccess ||
      (e = cudaMemcpy(ctx->d_W, c.W, w_bytes, cudaMemcpyHostToDevice)) != cudaSuccess ||
      (e = cudaMemcpy(ctx->d_b, bias.data(), n_b * 4, cudaMemcpyHostToDevice)) != cudaSuccess ||
      (e = cudaMemset(ctx->d_status, 0, 4)) != cudaSuccess) {
    free_ctx(ctx);
    return cuda_fail(e, "kvx_create: upload");
  }

  std::string why;
  ctx->tc_eligible = tc_supported(ctx, &why);
  ctx->xh_eligible = !ctx->tc_eligible && xh_supported(ctx, &why);
  ctx->F_xh = ctx->k * ctx->H * ctx->d;
  if (ctx->tc_eligible || ctx->xh_eligible) {
    // A per-head mapper with more selected layers than the per-head kernel holds in tensor
    // memory runs on the cross-head kernel: W of target head h widened to the cross-head
    // feature (every head of the k layers) with zeros outside head h's rows, which leaves
    // the map unchanged (the extra products are exact zeros).
    std::vector<uint8_t> wide;
    const void* w_xh = c.W;
    if (ctx->xh_eligible && ctx->head_mix == KVX_PER_HEAD) {
      const size_t es = ctx->weight_dtype == KVX_BF16 ? 2 : 4, d = ctx->d, F = ctx->F, Fx = ctx->F_xh;
      const size_t blocks = static_cast<size_t>(ctx->Lt) * 2 * ctx->H;
      wide.assign(blocks * Fx * d * es, 0);
      const uint8_t* w = static_cast<const uint8_t*>(c.W);
      for (size_t blk = 0; blk < blocks; ++blk) {
        const size_t h = blk % ctx->H;
        for (int j = 0; j < ctx->k; ++j)   // rows of selected layer j, head h: x = (j H + h) d
          std::memcpy(wide.data() + (blk * Fx + (j * ctx->H + h) * d) * d * es, w + (blk * F + j * d) * d * es,
                      d * d * es);
      }
      w_xh = wide.data();
    }
    kvx_status s = ctx->tc_eligible                  ? tc_prepare(ctx, c.W)
                   : ctx->weight_dtype == KVX_F32 ? repack_wt_hilo(ctx, w_xh, ctx->F_xh)
                                                  : repack_wt(ctx, w_xh, ctx->F_xh);
    if (s != KVX_OK) {
      free_ctx(ctx);
      return s;
    }
  }
  *out = ctx;
  return KVX_OK;
}

kvx_status kvx_destroy(kvx_ctx* ctx) {
  g_last_error.clear();
  if (!ctx) return KVX_OK;
  {
    DeviceGuard guard(ctx->device);
    cudaDeviceSynchronize();
  }
  free_ctx(ctx);
  return KVX_OK;
}

kvx_status kvx_get_selection(const kvx_ctx* ctx, int32_t* out) {
  g_last_error.clear();
  if (!ctx || !out) return fail(KVX_ERR_INVALID_ARG, "kvx_get_selection: NULL pointer");
  std::copy(ctx->sel.begin(), ctx->sel.end(), out);
  return KVX_OK;
}

kvx_status kvx_set_kernel(kvx_ctx* ctx, int32_t kernel) {
  g_last_error.clear();
  if (!ctx) return fail(KVX_ERR_INVALID_ARG, "kvx_set_kernel: NULL ctx");
  if (kernel != KVX_KERNEL_AUTO && kernel != KVX_KERNEL_SIMT && kernel != KVX_KERNEL_TCGEN05)
    return fail(KVX_ERR_INVALID_ARG, "kvx_set_kernel: unknown kernel");
  if (kernel == KVX_KERNEL_TCGEN05 && !ctx->tc_eligible && !ctx->xh_eligible) {
    std::string why;
    if (ctx->head_mix == KVX_CROSS_HEAD) xh_supported(ctx, &why); else tc_supported(ctx, &why);
    return fail(KVX_ERR_UNSUPPORTED, "kvx_set_kernel: tensor-core kernel unavailable: " + why);
  }
  ctx->kernel = kernel;
  return KVX_OK;
}

kvx_status kvx_get_kernel(const kvx_ctx* ctx, int32_t paged, int32_t* out) {
  g_last_error.clear();
  if (!ctx || !out) return fail(KVX_ERR_INVALID_ARG, "kvx_get_kernel: NULL argument");
  (void)paged;   // every kernel writes both target kinds
  if (ctx->xh_eligible && ctx->kernel != KVX_KERNEL_SIMT) *out = 3;
  else if (ctx->tc_eligible && ctx->kernel != KVX_KERNEL_SIMT) *out = 2;
  else *out = 1;
  return KVX_OK;
}

kvx_status kvx_set_test_wait(kvx_ctx* ctx, uint64_t wait_limit_ns, int64_t skip_bias_row) {
  g_last_error.clear();
  if (!ctx) return fail(KVX_ERR_INVALID_ARG, "kvx_set_test_wait: NULL ctx");
  if (wait_limit_ns != 0 && (wait_limit_ns < 1000000ull || wait_limit_ns > 4000000000ull))
    return fail(KVX_ERR_INVALID_ARG, "kvx_set_test_wait: wait limit outside [1 ms, 4 s]");
  if (skip_bias_row < -1 || skip_bias_row > INT32_MAX)
    return fail(KVX_ERR_INVALID_ARG, "kvx_set_test_wait: skip_bias_row must be -1 or a row index");
  ctx->wait_limit_ns = wait_limit_ns;
  ctx->skip_bias_row = skip_bias_row;
  return KVX_OK;
}

kvx_status kvx_get_status(kvx_ctx* ctx, void* stream) {
  g_last_error.clear();
  if (!ctx) return fail(KVX_ERR_INVALID_ARG, "kvx_get_status: NULL ctx");
  DeviceGuard guard(ctx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e, "kvx_get_status: stream sync");
  int32_t v = 0;
  if ((e = cudaMemcpy(&v, ctx->d_status, 4, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "kvx_get_status: read");
  if ((e = cudaMemset(ctx->d_status, 0, 4)) != cudaSuccess)
    return cuda_fail(e, "kvx_get_status: reset");
  if (v != KVX_OK) set_error(std::string("device reported ") + kvx_status_string((kvx_status)v));
  return static_cast<kvx_status>(v);
}

kvx_status kvx_map(kvx_ctx* ctx, const kvx_src* src, int32_t batch, int32_t tokens_per_seq,
                   const int32_t* positions, const kvx_tgt* tgt, void* stream) {
  NvtxRange range("kvx_map");
  g_last_error.clear();
  if (!ctx || !src || !tgt) return fail(KVX_ERR_INVALID_ARG, "kvx_map: NULL ctx/src/tgt");
  if (batch < 0 || tokens_per_seq < 0)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map: negative batch or tokens_per_seq");
  if (batch == 0 || tokens_per_seq == 0) return KVX_OK;
  if (!src->k || !src->v || !tgt->k || !tgt->v || !positions)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map: NULL cache or positions pointer");
  if (!aligned16(src->k) || !aligned16(src->v) || !aligned16(tgt->k) || !aligned16(tgt->v))
    return fail(KVX_ERR_INVALID_ARG, "kvx_map: cache pointers must be 16-byte aligned");
  if ((reinterpret_cast<uintptr_t>(positions) & 3u) != 0)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map: positions must be 4-byte aligned");
  for (int i = 0; i < 4; ++i)
    if (src->stride[i] < 0 || tgt->stride[i] < 0 || src->stride[i] % 8 != 0 || tgt->stride[i] % 8 != 0)
      return fail(KVX_ERR_INVALID_ARG,
                  "kvx_map: strides must be non-negative multiples of 8 elements");
  // head_dim contiguous: rows must not overlap within a (layer, head)
  if (src->stride[3] < ctx->d || tgt->stride[3] < ctx->d)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map: token stride smaller than head_dim");
  if (tgt->paged != 0 && tgt->paged != 1) return fail(KVX_ERR_INVALID_ARG, "kvx_map: paged must be 0 or 1");
  if (tgt->paged) {
    if (tgt->block_size <= 0 || !tgt->block_table || tgt->max_blocks_per_seq <= 0 || tgt->n_blocks <= 0)
      return fail(KVX_ERR_INVALID_ARG, "kvx_map: paged target needs block_size, block_table, "
                                       "max_blocks_per_seq and n_blocks > 0");
    if ((reinterpret_cast<uintptr_t>(tgt->block_table) & 3u) != 0)
      return fail(KVX_ERR_INVALID_ARG, "kvx_map: block_table must be 4-byte aligned");
  }
  MapArgs a{};
  a.src_k = src->k;
  a.src_v = src->v;
  a.tgt_k = tgt->k;
  a.tgt_v = tgt->v;
  for (int i = 0; i < 4; ++i) {
    a.ss[i] = src->stride[i];
    a.ts[i] = tgt->stride[i];
  }
  a.paged = tgt->paged;
  a.block_size = tgt->paged ? tgt->block_size : 1;
  a.max_blocks = tgt->paged ? tgt->max_blocks_per_seq : 0;
  a.n_blocks = tgt->paged ? tgt->n_blocks : 0;
  a.block_table = tgt->paged ? tgt->block_table : nullptr;
  a.pos = positions;
  a.B = batch;
  a.T = tokens_per_seq;

  DeviceGuard guard(ctx->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "kvx_map: cudaSetDevice");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // cross-head: the tensor-core kernel writes contiguous and paged targets
  if (ctx->xh_eligible && ctx->kernel != KVX_KERNEL_SIMT) return launch_xh(ctx, a, st);
  const bool use_tc = ctx->kernel == KVX_KERNEL_TCGEN05 || (ctx->kernel == KVX_KERNEL_AUTO && ctx->tc_eligible);
  return use_tc ? launch_tc(ctx, a, st) : launch_simt(ctx, a, st);
}

}  // extern "C"
