// Mapping caches that live in host memory: the tokens are cut into chunks and three
// streams overlap the host-to-device copy of chunk c+1, the map of chunk c and the
// device-to-host copy of chunk c-1 (two staging slots per buffer, ordered by events).
// GB300's host link carries about 200 GB/s each way and ~340 GB/s both ways at once, so a
// step that moves the source in and the targets out is bounded by the larger of the two
// copies rather than by their sum plus the map.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <string>

#include "kvx_internal.h"

struct kvx_host_pipe {
  kvx_ctx* ctx = nullptr;
  int device = 0;
  int32_t B = 0, chunk = 0;
  size_t esz = 0;                       // bytes per cache element
  cudaStream_t s_h2d = nullptr, s_comp = nullptr, s_d2h = nullptr;
  cudaEvent_t ev_start = nullptr;
  cudaEvent_t ev_h2d[2] = {nullptr, nullptr}, ev_map[2] = {nullptr, nullptr}, ev_d2h[2] = {nullptr, nullptr};
  bool used[2] = {false, false};
  char* mem = nullptr;                  // one device allocation for every staging buffer
  char* src_k[2] = {nullptr, nullptr};
  char* src_v[2] = {nullptr, nullptr};
  char* tgt_k[2] = {nullptr, nullptr};
  char* tgt_v[2] = {nullptr, nullptr};
  int32_t* pos[2] = {nullptr, nullptr};
};

namespace {

kvx_status pipe_fail(kvx_status s, const std::string& m) {
  kvx::set_error(m);
  return s;
}

void release(kvx_host_pipe* p) {
  if (!p) return;
  int prev = 0;
  cudaGetDevice(&prev);
  cudaSetDevice(p->device);
  for (cudaStream_t s : {p->s_h2d, p->s_comp, p->s_d2h})
    if (s) cudaStreamSynchronize(s);
  for (cudaStream_t s : {p->s_h2d, p->s_comp, p->s_d2h})
    if (s) cudaStreamDestroy(s);
  if (p->ev_start) cudaEventDestroy(p->ev_start);
  for (int i = 0; i < 2; ++i)
    for (cudaEvent_t e : {p->ev_h2d[i], p->ev_map[i], p->ev_d2h[i]})
      if (e) cudaEventDestroy(e);
  cudaFree(p->mem);
  cudaSetDevice(prev);
  delete p;
}

// Host caches must be contiguous [L][B][H][T][d]: element (l, b, h, t, c) at
// (((l B + b) H + h) T + t) d + c.
bool contiguous(const int64_t* s, int32_t B, int32_t H, int32_t T, int32_t d) {
  return s[3] == d && s[2] == static_cast<int64_t>(T) * d && s[1] == static_cast<int64_t>(H) * s[2] &&
         s[0] == static_cast<int64_t>(B) * s[1];
}

}  // namespace

extern "C" {

KVX_API kvx_status kvx_host_pipe_create(kvx_ctx* ctx, int32_t batch, int32_t chunk_tokens, kvx_host_pipe** out) {
  kvx::set_error("");
  if (!out) return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_host_pipe_create: out is NULL");
  *out = nullptr;
  if (!ctx) return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_host_pipe_create: NULL ctx");
  if (batch < 1 || chunk_tokens < 1)
    return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_host_pipe_create: batch and chunk_tokens must be >= 1");
  auto* p = new kvx_host_pipe;
  p->ctx = ctx;
  p->device = ctx->device;
  p->B = batch;
  p->chunk = chunk_tokens;
  p->esz = ctx->cache_dtype == KVX_F32 ? 4 : 2;
  int prev = 0;
  cudaGetDevice(&prev);
  cudaError_t e = cudaSetDevice(p->device);
  const size_t row = static_cast<size_t>(batch) * ctx->H * chunk_tokens * ctx->d * p->esz;   // one layer
  const size_t src_b = static_cast<size_t>(ctx->Ls) * row, tgt_b = static_cast<size_t>(ctx->Lt) * row;
  const size_t pos_b = (static_cast<size_t>(batch) * chunk_tokens * 4 + 255) / 256 * 256;
  const size_t slot = 2 * src_b + 2 * tgt_b + pos_b;
  if (e == cudaSuccess) e = cudaMalloc(&p->mem, 2 * slot);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p->s_h2d, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p->s_comp, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p->s_d2h, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->ev_start, cudaEventDisableTiming);
  for (int i = 0; i < 2 && e == cudaSuccess; ++i) {
    e = cudaEventCreateWithFlags(&p->ev_h2d[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->ev_map[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->ev_d2h[i], cudaEventDisableTiming);
    if (e == cudaSuccess) {
      char* b = p->mem + i * slot;
      p->src_k[i] = b;
      p->src_v[i] = b + src_b;
      p->tgt_k[i] = b + 2 * src_b;
      p->tgt_v[i] = b + 2 * src_b + tgt_b;
      p->pos[i] = reinterpret_cast<int32_t*>(b + 2 * src_b + 2 * tgt_b);
    }
  }
  cudaSetDevice(prev);
  if (e != cudaSuccess) {
    const kvx_status s = e == cudaErrorMemoryAllocation ? KVX_ERR_OOM : KVX_ERR_CUDA;
    release(p);
    return pipe_fail(s, std::string("kvx_host_pipe_create: ") + cudaGetErrorString(e));
  }
  *out = p;
  return KVX_OK;
}

KVX_API kvx_status kvx_map_host(kvx_host_pipe* p, const kvx_src* src, int32_t tokens_per_seq, const int32_t* positions,
                                const kvx_tgt* tgt, void* stream) {
  kvx::NvtxRange range("kvx_map_host");
  kvx::set_error("");
  if (!p || !src || !tgt || !positions) return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_map_host: NULL argument");
  if (tokens_per_seq < 0) return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_map_host: negative tokens_per_seq");
  if (tokens_per_seq == 0) return KVX_OK;
  const kvx_ctx* c = p->ctx;
  if (!src->k || !src->v || !tgt->k || !tgt->v) return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_map_host: NULL cache pointer");
  if (tgt->paged) return pipe_fail(KVX_ERR_UNSUPPORTED, "kvx_map_host: host targets must be contiguous");
  const int32_t T = tokens_per_seq, B = p->B;
  if (!contiguous(src->stride, B, c->H, T, c->d) || !contiguous(tgt->stride, B, c->H, T, c->d))
    return pipe_fail(KVX_ERR_INVALID_ARG, "kvx_map_host: host caches must be contiguous [L][B][H][T][d]");
  int prev = 0;
  cudaGetDevice(&prev);
  cudaError_t e = cudaSetDevice(p->device);
  const cudaStream_t caller = static_cast<cudaStream_t>(stream);
  const size_t d_b = static_cast<size_t>(c->d) * p->esz;           // one token row of one head
  const size_t spitch = static_cast<size_t>(T) * d_b, stg_pitch = static_cast<size_t>(p->chunk) * d_b;
  const size_t src_rows = static_cast<size_t>(c->Ls) * B * c->H, tgt_rows = static_cast<size_t>(c->Lt) * B * c->H;
  kvx_status result = KVX_OK;
  if (e == cudaSuccess) e = cudaEventRecord(p->ev_start, caller);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_h2d, p->ev_start, 0);
  int last = 0;
  for (int32_t t0 = 0, ch = 0; t0 < T && e == cudaSuccess && result == KVX_OK; t0 += p->chunk, ++ch) {
    const int s = ch & 1;
    last = s;
    const int32_t n = std::min(p->chunk, T - t0);
    // 1. host -> device (the slot's previous map must have read it)
    if (p->used[s]) e = cudaStreamWaitEvent(p->s_h2d, p->ev_map[s], 0);
    const char* hk = static_cast<const char*>(src->k) + t0 * d_b;
    const char* hv = static_cast<const char*>(src->v) + t0 * d_b;
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(p->src_k[s], stg_pitch, hk, spitch, n * d_b, src_rows, cudaMemcpyHostToDevice, p->s_h2d);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(p->src_v[s], stg_pitch, hv, spitch, n * d_b, src_rows, cudaMemcpyHostToDevice, p->s_h2d);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(p->pos[s], static_cast<size_t>(n) * 4, positions + t0, static_cast<size_t>(T) * 4,
                            static_cast<size_t>(n) * 4, B, cudaMemcpyHostToDevice, p->s_h2d);
    if (e == cudaSuccess) e = cudaEventRecord(p->ev_h2d[s], p->s_h2d);
    // 2. the map of the chunk (the slot's targets must have gone out)
    if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_comp, p->ev_h2d[s], 0);
    if (e == cudaSuccess && p->used[s]) e = cudaStreamWaitEvent(p->s_comp, p->ev_d2h[s], 0);
    if (e != cudaSuccess) break;
    kvx_src ss{};
    ss.k = p->src_k[s];
    ss.v = p->src_v[s];
    ss.stride[3] = c->d;
    ss.stride[2] = static_cast<int64_t>(p->chunk) * c->d;
    ss.stride[1] = static_cast<int64_t>(c->H) * ss.stride[2];
    ss.stride[0] = static_cast<int64_t>(B) * ss.stride[1];
    kvx_tgt ts{};
    ts.k = p->tgt_k[s];
    ts.v = p->tgt_v[s];
    for (int i = 0; i < 4; ++i) ts.stride[i] = ss.stride[i];
    result = kvx_map(p->ctx, &ss, B, n, p->pos[s], &ts, p->s_comp);
    if (result != KVX_OK) break;
    e = cudaEventRecord(p->ev_map[s], p->s_comp);
    // 3. device -> host
    if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_d2h, p->ev_map[s], 0);
    char* ok = static_cast<char*>(tgt->k) + t0 * d_b;
    char* ov = static_cast<char*>(tgt->v) + t0 * d_b;
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(ok, spitch, p->tgt_k[s], stg_pitch, n * d_b, tgt_rows, cudaMemcpyDeviceToHost, p->s_d2h);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(ov, spitch, p->tgt_v[s], stg_pitch, n * d_b, tgt_rows, cudaMemcpyDeviceToHost, p->s_d2h);
    if (e == cudaSuccess) e = cudaEventRecord(p->ev_d2h[s], p->s_d2h);
    p->used[s] = true;
  }
  // the caller's stream resumes once every chunk is back in host memory
  if (e == cudaSuccess && result == KVX_OK) e = cudaStreamWaitEvent(caller, p->ev_d2h[last], 0);
  cudaSetDevice(prev);
  if (result != KVX_OK) return result;
  if (e != cudaSuccess) return pipe_fail(KVX_ERR_CUDA, std::string("kvx_map_host: ") + cudaGetErrorString(e));
  return KVX_OK;
}

KVX_API kvx_status kvx_host_pipe_destroy(kvx_host_pipe* p) {
  release(p);
  return KVX_OK;
}

}  // extern "C"
