// kvx_map_noalloc: the SIMT mapping kernel run without any allocation by the library,
// for callers that cannot let a library call cudaMalloc (see include/kvx.h).  The paper
// has no counterpart; the computation is the one kvx_map performs with KVX_KERNEL_SIMT.
//
// The only device memory used besides the caller's buffers is g_noalloc_scratch, a
// file-scope array every GPU holds from library load to process exit:
//   bytes [0, 4)                    device status word (cleared by every call)
//   bytes [256, 256 + 4 * L_t * k)  copy of the selection table (rewritten by every call)
// All calls on a device share it, so calls that overlap on the GPU race on it.
#include <algorithm>
#include <cmath>
#include <mutex>
#include <string>

#include "kvx_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[KVX_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_addr_mutex;
void* g_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on `device` (the caller has made it current).
// Looked up once per device; host code may not use the symbol's name as an address.
kvx_status scratch_address(int device, unsigned char** out) {
  if (device < 0 || device >= kMaxDevices) {
    kvx::set_error("kvx_map_noalloc: device index out of range");
    return KVX_ERR_INVALID_ARG;
  }
  std::lock_guard<std::mutex> lock(g_addr_mutex);
  if (!g_addr[device]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) {
      kvx::set_error(std::string("kvx_map_noalloc: cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      return KVX_ERR_CUDA;
    }
    g_addr[device] = p;
  }
  *out = static_cast<unsigned char*>(g_addr[device]);
  return KVX_OK;
}

kvx_status fail(kvx_status s, const char* msg) {
  kvx::set_error(msg);
  return s;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

}  // namespace

extern "C" KVX_API kvx_status kvx_map_noalloc(const kvx_noalloc_mapper* m, int device, const kvx_src* src,
                                              int32_t batch, int32_t tokens_per_seq, const int32_t* positions,
                                              const kvx_tgt* tgt, void* stream, int32_t* device_status) {
  kvx::set_error("");
  if (!m || !src || !tgt) return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: NULL mapper/src/tgt");
  if (m->src_layers <= 0 || m->tgt_layers <= 0 || m->n_kv_heads <= 0 || m->head_dim <= 0 ||
      m->head_dim % 2 != 0 || m->head_dim > kvx::kMaxHeadDim)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: bad layer/head/head_dim counts");
  if (m->k < 1 || m->k > m->src_layers) return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: k outside [1, src_layers]");
  if (static_cast<int64_t>(m->tgt_layers) * m->k > KVX_NOALLOC_MAX_SELECTION)
    return fail(KVX_ERR_INVALID_ARG,
                "kvx_map_noalloc: tgt_layers * k exceeds KVX_NOALLOC_MAX_SELECTION (16384)");
  if ((m->rope_style != KVX_ROPE_HALF && m->rope_style != KVX_ROPE_INTERLEAVED) ||
      (m->cache_dtype != KVX_F32 && m->cache_dtype != KVX_BF16) ||
      (m->weight_dtype != KVX_F32 && m->weight_dtype != KVX_BF16) ||
      (m->head_mix != KVX_PER_HEAD && m->head_mix != KVX_CROSS_HEAD) || m->reserved != 0)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: bad rope_style, dtype, head_mix or reserved");
  if (!(m->src_rope_theta > 1.0) || !(m->tgt_rope_theta > 1.0) || !std::isfinite(m->src_rope_theta) ||
      !std::isfinite(m->tgt_rope_theta))
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: rope thetas must be finite and > 1");
  if (const char* why = kvx::check_rope_scaling(m->src_rope_scaling))
    return fail(KVX_ERR_INVALID_ARG, (std::string("kvx_map_noalloc: source ") + why).c_str());
  if (const char* why = kvx::check_rope_scaling(m->tgt_rope_scaling))
    return fail(KVX_ERR_INVALID_ARG, (std::string("kvx_map_noalloc: target ") + why).c_str());
  if (!m->selection || !m->W || !m->b) return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: NULL selection, W or b");
  if (!aligned(m->W, 16) || !aligned(m->b, 16))
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: W and b must be 16-byte aligned");
  if (m->rope_numerics != KVX_ROPE_EXACT && m->rope_numerics != KVX_ROPE_HF)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: bad rope_numerics");
  for (int64_t i = 0; i < static_cast<int64_t>(m->tgt_layers) * m->k; ++i)
    if (m->selection[i] < 0 || m->selection[i] >= m->src_layers)
      return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: selection entry outside [0, src_layers)");
  for (int64_t l = 0; l < m->tgt_layers; ++l) {  // a row names k distinct source layers
    const int32_t* row = m->selection + l * m->k;
    for (int i = 0; i < m->k; ++i)
      for (int j = 0; j < i; ++j)
        if (row[i] == row[j])
          return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: duplicate source layer in a selection row");
  }
  if (batch < 0 || tokens_per_seq < 0) return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: negative sizes");
  if (device_status) *device_status = KVX_OK;
  if (batch == 0 || tokens_per_seq == 0) return KVX_OK;
  if (!src->k || !src->v || !tgt->k || !tgt->v || !positions)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: NULL cache or positions pointer");
  if (!aligned(src->k, 16) || !aligned(src->v, 16) || !aligned(tgt->k, 16) || !aligned(tgt->v, 16) ||
      !aligned(positions, 4))
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: misaligned cache or positions pointer");
  for (int i = 0; i < 4; ++i)
    if (src->stride[i] < 0 || tgt->stride[i] < 0 || src->stride[i] % 8 != 0 || tgt->stride[i] % 8 != 0)
      return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: strides must be non-negative multiples of 8 elements");
  if (src->stride[3] < m->head_dim || tgt->stride[3] < m->head_dim)
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: token stride smaller than head_dim");
  if (tgt->paged != 0 && tgt->paged != 1) return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: paged must be 0 or 1");
  if (tgt->paged && (tgt->block_size <= 0 || !tgt->block_table || tgt->max_blocks_per_seq <= 0 ||
                     tgt->n_blocks <= 0 || !aligned(tgt->block_table, 4)))
    return fail(KVX_ERR_INVALID_ARG, "kvx_map_noalloc: bad paged target description");

  int prev = -1;
  cudaError_t e = cudaGetDevice(&prev);
  if (e == cudaSuccess && prev != device) e = cudaSetDevice(device);
  if (e != cudaSuccess) return fail(KVX_ERR_CUDA, "kvx_map_noalloc: cudaSetDevice failed");
  struct Restore {
    int prev, dev;
    ~Restore() {
      if (prev >= 0 && prev != dev) cudaSetDevice(prev);
    }
  } restore{prev, device};

  unsigned char* scratch = nullptr;
  kvx_status st = scratch_address(device, &scratch);
  if (st != KVX_OK) return st;
  int32_t* d_status = reinterpret_cast<int32_t*>(scratch);
  int32_t* d_sel = reinterpret_cast<int32_t*>(scratch + 256);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t sel_bytes = static_cast<size_t>(m->tgt_layers) * m->k * 4;
  if ((e = cudaMemsetAsync(d_status, 0, 4, s)) != cudaSuccess ||
      (e = cudaMemcpyAsync(d_sel, m->selection, sel_bytes, cudaMemcpyHostToDevice, s)) != cudaSuccess)
    return fail(KVX_ERR_CUDA, "kvx_map_noalloc: staging the status word or selection failed");

  // A host-side description of the mapper pointing at the caller's buffers and the
  // scratch array; nothing here owns device memory.
  kvx_ctx view;
  view.device = device;
  view.Ls = m->src_layers;
  view.Lt = m->tgt_layers;
  view.H = m->n_kv_heads;
  view.d = m->head_dim;
  view.k = m->k;
  view.head_mix = m->head_mix;
  view.F = m->k * m->head_dim * (m->head_mix == KVX_CROSS_HEAD ? m->n_kv_heads : 1);
  view.rope_style = m->rope_style;
  view.cache_dtype = m->cache_dtype;
  view.weight_dtype = m->weight_dtype;
  view.theta_s = m->src_rope_theta;
  view.theta_t = m->tgt_rope_theta;
  view.rope_numerics = m->rope_numerics;
  kvx::set_rope_scaling(&view, m->src_rope_scaling, m->tgt_rope_scaling);
  kvx::fill_rope(&view);
  view.d_sel = d_sel;
  view.d_W = const_cast<void*>(m->W);
  view.d_b = const_cast<float*>(m->b);
  view.d_status = d_status;

  kvx::MapArgs a{};
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
  st = kvx::launch_simt(&view, a, s);  // the view only borrows these pointers
  if (st != KVX_OK) return st;
  if (device_status) {
    int32_t v = 0;
    if ((e = cudaMemcpyAsync(&v, d_status, 4, cudaMemcpyDeviceToHost, s)) != cudaSuccess ||
        (e = cudaStreamSynchronize(s)) != cudaSuccess)
      return fail(KVX_ERR_CUDA, "kvx_map_noalloc: reading the device status failed");
    *device_status = v;
  }
  return KVX_OK;
}
