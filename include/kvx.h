/*
 * kvx -- cross-model KV-cache mapper, GB300 (sm_103a) C ABI.
 *
 * Applies the closed-form per-head ridge mapper of "Cross-Model KV Cache Transfer in
 * LLM Families: A Closed-Form Linear Mapping for Prefill Reuse" (arXiv 2608.03893) to
 * a prefilled source KV cache and writes the target model's KV cache:
 *
 *   for every target layer l, KV head h and token with absolute position t
 *     X_K = [ R_s(t)^-1 K_s^{sel[l][0]}[h] || ... || R_s(t)^-1 K_s^{sel[l][k-1]}[h] ]
 *     X_V = [ V_s^{sel[l][0]}[h]           || ... || V_s^{sel[l][k-1]}[h] ]
 *     K_t^l[h] = R_t(t) (X_K W_K^{l,h} + b_K^{l,h})          (Sec. 3.3 composition)
 *     V_t^l[h] =         X_V W_V^{l,h} + b_V^{l,h}            (Eq. ridge_kv, Sec. 3.1)
 *
 * sel[l] are the top-k source layers of target layer l (Sec. 3.2); R_theta(t) is the
 * RoPE rotation of pair i by t * theta^(-2i/d) (Sec. 3.3); source and target tokens
 * share the absolute position t (Sec. 3.3).  X is a row vector (Sec. 2.3, Eq.
 * single_source_ols).  For bf16 caches the stripped keys are rounded to bf16
 * (round-to-nearest-even) before the contraction: the one operand a bf16 forward
 * (Appendix "Run information", precision row) materialises; the contraction
 * accumulates in fp32 and the output is rounded once to the cache dtype.
 *
 * Conventions for every call:
 *  - No call throws; every call returns a kvx_status (or a documented value).
 *  - Device pointers must be 16-byte aligned, caches must have head_dim contiguous,
 *    and every other stride must be a multiple of 8 elements (16 bytes for bf16).
 *  - A kvx_ctx must not be used from two host threads at once, nor mapped on two
 *    streams at the same time (both launches share the context's status word).
 *  - kvx_last_error() returns a thread-local, human-readable description of the last
 *    non-OK status returned on the calling thread.
 */
#ifndef KVX_H
#define KVX_H

#include <stdint.h>

#if defined(__GNUC__)
#define KVX_API __attribute__((visibility("default")))
#else
#define KVX_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct kvx_ctx kvx_ctx;

typedef enum {
  KVX_OK = 0,
  KVX_ERR_INVALID_ARG = 1,   /* a bad argument, detected on the host; nothing launched */
  KVX_ERR_UNSUPPORTED = 2,   /* valid request that the library cannot run (e.g. shape) */
  KVX_ERR_OOM = 3,           /* cudaMalloc failed in kvx_create */
  KVX_ERR_CUDA = 4,          /* a CUDA runtime or launch error */
  KVX_ERR_TIMEOUT = 5,       /* device: a bounded wait in a kernel ran out */
  KVX_ERR_DEVICE_BOUNDS = 6  /* device: position < 0 or block-table entry outside the pool */
} kvx_status;

typedef enum { KVX_F32 = 0, KVX_BF16 = 1 } kvx_dtype;

/* Pair layout of the RoPE rotation (the paper does not state one).
 * HALF: pairs (i, i + d/2) (Qwen3 / Llama checkpoints).  INTERLEAVED: pairs (2i, 2i+1). */
typedef enum { KVX_ROPE_HALF = 0, KVX_ROPE_INTERLEAVED = 1 } kvx_rope_style;

/* Feature layout.  PER_HEAD: head h of the k selected layers, F = k * head_dim.
 * CROSS_HEAD: all KV heads of the k selected layers, head-minor, F = k * n_kv * head_dim
 * (the paper's d_s = k n_kv d_h, Sec. 3.1 / Sec. 3.2). */
typedef enum { KVX_PER_HEAD = 0, KVX_CROSS_HEAD = 1 } kvx_head_mix;

/* Which kernel kvx_map launches.  AUTO picks a tensor-core (tcgen05) kernel when the
 * shape allows it (bf16 caches, head_dim 128, HALF or INTERLEAVED pairs; PER_HEAD with
 * k <= 4 on the per-head kernel; CROSS_HEAD, and PER_HEAD with k > 4 on W widened with
 * zeros, on the cross-head kernel, which needs an even head count; contiguous or paged
 * targets) and the fp32 SIMT kernel otherwise.
 * fp32 weights run on the tensor cores split into bf16 hi = bf16(w) and lo = bf16(w - hi)
 * (twice the MMAs; the contraction follows the fp32 W to within 2^-17 of each weight).
 * The CROSS_HEAD tensor-core kernel keeps a workspace for the stripped source keys
 * (L_s * B * n_kv * T * head_dim bf16) in the context, allocated by the first
 * kvx_map that needs it (a blocking cudaMalloc) and grown when a later call needs more;
 * kvx_destroy frees it. */
typedef enum { KVX_KERNEL_AUTO = 0, KVX_KERNEL_SIMT = 1, KVX_KERNEL_TCGEN05 = 2 } kvx_kernel;

/* RoPE numerics.  EXACT: angles t omega_i to ~1e-6 rad and the rotations in fp32 (the
 * definition; the default).  HF: the rounding of the Hugging Face bf16 forward that wrote
 * the caches -- the angle is the fp32 product of fp32(t) and fp32(omega_i), cos and sin of
 * it are rounded to the cache dtype, and each product and sum of the rotation is rounded
 * to the cache dtype (x' = r(r(a c) + r(-b s)), y' = r(r(b c) + r(a s)); the strip uses -s);
 * the mapped keys are rounded to the cache dtype before the target rotation.  Every map
 * kernel, kvx_fit_ridge, kvx_r2_probe and kvx_mlp_map implement both. */
typedef enum { KVX_ROPE_EXACT = 0, KVX_ROPE_HF = 1 } kvx_rope_numerics;

/* Llama-3 RoPE frequency scaling (the rope_scaling of the Llama 3.1 checkpoints:
 * factor 8, low_freq_factor 1, high_freq_factor 4, original_max_position 8192).  With
 * omega_i = theta^(-2i/d) and wavelength 2 pi / omega_i: below original_max_position /
 * high_freq_factor omega_i is kept, above original_max_position / low_freq_factor it is
 * divided by factor, and in between it is (1 - s) omega_i / factor + s omega_i with
 * s = (original_max_position / wavelength - low_freq_factor) / (high_freq_factor -
 * low_freq_factor).  The paper uses Llama 3.1 pairs but does not discuss the scaling; a
 * NULL pointer below means plain theta.  factor >= 1, 0 < low < high, position > 0. */
typedef struct {
  double factor, low_freq_factor, high_freq_factor, original_max_position;
} kvx_rope_scaling;

/* Mapper description, read by kvx_create.  All pointers are HOST pointers; the
 * context copies what it needs, so they may be freed when kvx_create returns. */
typedef struct {
  int32_t src_layers;        /* L_s */
  int32_t tgt_layers;        /* L_t */
  int32_t n_kv_heads;        /* n_kv = n_kv^s = n_kv^t (matched KV, Sec. 2.1) */
  int32_t head_dim;          /* d = d_h^s = d_h^t, even */
  int32_t k;                 /* source layers per target layer, 1 <= k <= L_s */
  int32_t rope_style;        /* kvx_rope_style */
  double src_rope_theta;     /* Theta of the source model's RoPE */
  double tgt_rope_theta;     /* Theta of the target model's RoPE */
  int32_t cache_dtype;       /* kvx_dtype of the source and target caches */
  int32_t weight_dtype;      /* kvx_dtype of W and b below */
  int32_t head_mix;          /* kvx_head_mix */
  int32_t reserved;          /* must be 0 */
  /* [L_t][k] selected source layers, distinct, each in [0, L_s); row block j of W
   * belongs to selection[l][j].  NULL: take the top-k of selection_scores. */
  const int32_t* selection;
  /* [L_t][L_s] scores (head-averaged R^2, Sec. 3.2); used only if selection is NULL. */
  const double* selection_scores;
  /* [L_t][2][n_kv][F][d] in weight_dtype; index 0 of axis 1 is K, 1 is V. */
  const void* W;
  /* [L_t][2][n_kv][d] in weight_dtype, or NULL for a zero bias (Sec. 3.1: the
   * centred fit gives b = mean(Y) - mean(X) W*). */
  const void* b;
  /* RoPE frequency scaling of the source / target model, or NULL (plain theta). */
  const kvx_rope_scaling* src_rope_scaling;
  const kvx_rope_scaling* tgt_rope_scaling;
  int32_t rope_numerics;     /* kvx_rope_numerics */
} kvx_config;

/* Source cache, DEVICE memory owned by the caller: element (layer l, batch b, head h,
 * token t, channel c) of K (V) is at k[l*stride[0] + b*stride[1] + h*stride[2] +
 * t*stride[3] + c] (v[...]).  Strides in elements; K and V share them.  The keys are
 * the stored (RoPE-rotated) keys.  Must stay valid until the stream work completes. */
typedef struct {
  const void* k;
  const void* v;
  int64_t stride[4];
} kvx_src;

/* Target cache, DEVICE memory owned by the caller.
 * paged == 0 (contiguous): token t of sequence b goes to
 *   k[l*stride[0] + b*stride[1] + h*stride[2] + t*stride[3] + c].
 * paged == 1: the token at position p of sequence b goes to physical block
 *   blk = block_table[b * max_blocks_per_seq + p / block_size], slot p % block_size:
 *   k[l*stride[0] + blk*stride[1] + h*stride[2] + (p % block_size)*stride[3] + c].
 *   block_table is DEVICE int32 [batch][max_blocks_per_seq]; an entry outside
 *   [0, n_blocks) or a logical block >= max_blocks_per_seq sets KVX_ERR_DEVICE_BOUNDS
 *   in the status word and that row is not written.
 * Only the mapped tokens are written; every other element is left untouched, which is
 * what lets successive turns of a conversation append to one cache (Sec. 4.5). */
typedef struct {
  int32_t paged;
  int32_t block_size;
  void* k;
  void* v;
  int64_t stride[4];
  const int32_t* block_table;
  int32_t max_blocks_per_seq;
  int32_t n_blocks;
} kvx_tgt;

/* Build a mapper on CUDA device `device`: validates the configuration, takes the
 * selection (given, or the top-k of the scores, Sec. 3.2), and copies W and b to the
 * device in the kernels' layouts.  The context owns all of its device memory.
 * Errors: INVALID_ARG (bad dims, k, selection, NULL W), UNSUPPORTED (head_dim > 256 or
 * odd), OOM, CUDA.  On error *out is set to NULL. */
KVX_API kvx_status kvx_create(const kvx_config* cfg, int device, kvx_ctx** out);

/* Map `batch` sequences of `tokens_per_seq` tokens each (Eq. ridge_kv with the Sec. 3.3
 * RoPE composition).  positions: DEVICE int32 [batch][tokens_per_seq], the absolute
 * position of each token, shared by source and target (Sec. 3.3); for a contiguous
 * target the token index t also addresses the output row.  Asynchronous on `stream`
 * (a cudaStream_t; NULL = the legacy default stream).  Host-detected errors return
 * before any launch (INVALID_ARG, UNSUPPORTED); launch failures return CUDA;
 * device-detected errors go to the status word read by kvx_get_status.
 * batch == 0 or tokens_per_seq == 0 is a no-op returning OK.
 * kvx_map may be captured into a CUDA graph: it only encodes tensor maps on the host and
 * launches (the cross-head kernel's workspace is allocated by the first call that needs
 * it, so make one call of the captured shape before the capture); a replay maps whatever
 * the captured buffers then hold. */
KVX_API kvx_status kvx_map(kvx_ctx* ctx, const kvx_src* src, int32_t batch, int32_t tokens_per_seq,
                   const int32_t* positions, const kvx_tgt* tgt, void* stream);

/* ---- Mapping caches in host memory, copies overlapped with the map ---------------
 * A pipe holds device staging for `chunk_tokens` tokens of `batch` sequences (two slots
 * of source K, V, positions and target K, V: about 4 chunk_tokens batch n_kv d (L_s + L_t)
 * cache elements) and three internal streams.  kvx_map_host maps host caches through it:
 * the tokens go in chunks, and the host-to-device copy of one chunk, the map of the
 * previous one and the device-to-host copy of the one before run at the same time.  The
 * results equal kvx_map's on device copies of the same caches.
 * Host layouts: src contiguous [L_s][batch][n_kv][T][d] (stride = {batch n_kv T d,
 * n_kv T d, T d, d}), tgt contiguous [L_t][batch][n_kv][T][d] (paged: UNSUPPORTED),
 * positions [batch][T]; pinned memory (cudaHostAlloc / cudaHostRegister) for the copies
 * to overlap.  The work starts after the work already queued on `stream` and `stream`
 * waits for its end, so the host targets are complete once `stream` is; the host inputs
 * must not change until then.  Device errors go to the context's status word
 * (kvx_get_status).  A pipe serves one caller at a time; destroy it before its context. */
typedef struct kvx_host_pipe kvx_host_pipe;
KVX_API kvx_status kvx_host_pipe_create(kvx_ctx* ctx, int32_t batch, int32_t chunk_tokens, kvx_host_pipe** out);
KVX_API kvx_status kvx_map_host(kvx_host_pipe* pipe, const kvx_src* src, int32_t tokens_per_seq,
                                const int32_t* positions, const kvx_tgt* tgt, void* stream);
KVX_API kvx_status kvx_host_pipe_destroy(kvx_host_pipe* pipe);

/* Free the context and its device memory (synchronises the device first). NULL is OK. */
KVX_API kvx_status kvx_destroy(kvx_ctx* ctx);

/* Top-k source-layer selection (Sec. 3.2), on the host: for each target layer the k
 * highest scores; ties go to the lower source index; each row of out[L_t][k] is
 * returned in ascending source-layer order.  INVALID_ARG for NULL or k outside
 * [1, L_s]. */
KVX_API kvx_status kvx_select_topk(const double* scores, int32_t tgt_layers, int32_t src_layers,
                           int32_t k, int32_t* out);

/* The per-head tensor-core kernel's source-tile load schedule for a selection table, as
 * kvx_create builds it (host only; no device needed).  The gather of Sec. 3.2 reads
 * source layers selection[l][0..k-1] for every target layer l; the kernel keeps up to
 * four source tiles of a token tile in tensor memory and loads each tile when a use
 * needs it, evicting the resident tile whose next use is farthest away (Belady), so a
 * layer shared by consecutive target layers is read from HBM once per token tile.
 *   selection   host int32 [L_t][k] (row l: distinct layers in [0, L_s)), caller-owned
 *   n_loads     out: source-tile loads per token tile (≤ L_t·k)
 *   load_layer  out int32 [L_t·k]: the source layer of load e (first *n_loads valid)
 *   load_word   out int32 [L_t·k]: bits 0-1 the slot of load e; bit 2 + i set if issuer i
 *               (issuer of the target layers l with l % 2 == i) must release the slot's
 *               previous tile before load e (for the slot's first load of a token tile:
 *               the last tile of the previous token tile); bit 4 + i set if issuer i uses
 *               the loaded tile
 *   use_word    out int32 [L_t·k]: for use (l, j) at l·k + j, bits 0-1 the slot it reads;
 *               bit 2 set on the issuer's first use of the tile (it waits for the load);
 *               bit 4 set on its last use (it releases the slot after the use)
 * INVALID_ARG for a NULL pointer, sizes below 1, k > L_s, an entry out of range or a
 * repeated layer in a row; UNSUPPORTED for k > 4.  No state is kept. */
KVX_API kvx_status kvx_tc_load_schedule(const int32_t* selection, int32_t src_layers, int32_t tgt_layers,
                                        int32_t k, int32_t* n_loads, int32_t* load_layer, int32_t* load_word,
                                        int32_t* use_word);

/* Copy the context's selection table to host out[L_t][k]. */
KVX_API kvx_status kvx_get_selection(const kvx_ctx* ctx, int32_t* out);

/* Choose the kernel for later kvx_map calls (kvx_kernel).  UNSUPPORTED if the
 * configuration cannot run on the requested kernel. */
KVX_API kvx_status kvx_set_kernel(kvx_ctx* ctx, int32_t kernel);

/* Which kernel kvx_map runs on ctx for a contiguous (paged = 0) or paged (paged = 1)
 * target under the current kvx_set_kernel choice: *out = 1 the fp32 SIMT kernel, 2 the
 * per-head tensor-core kernel (one launch), 3 the cross-head tensor-core kernel (a key-strip
 * launch and a GEMM launch; per-head mappers with k > 4 run here on W widened with zeros
 * outside each head's rows).  INVALID_ARG for a NULL argument. */
KVX_API kvx_status kvx_get_kernel(const kvx_ctx* ctx, int32_t paged, int32_t* out);

/* Synchronise `stream`, return the device status word (KVX_OK or the first
 * device-detected error since the last call) and reset it to KVX_OK. */
KVX_API kvx_status kvx_get_status(kvx_ctx* ctx, void* stream);

/* Test switch of the bounded waits (the paper has no counterpart).  Every wait of the
 * per-head tensor-core kernel gives up after 4 s, sets KVX_ERR_TIMEOUT in the status word
 * and makes the kernel drain its copies and MMAs in flight, free its tensor memory and
 * return.  A test exercises that path on a healthy GPU with this call:
 *   wait_limit_ns  the bound of every wait of later kvx_map calls on ctx, in [1 ms, 4 s],
 *                  or 0 for the default 4 s;
 *   skip_bias_row  >= 0: the first CTA of later launches never loads its bias row of this
 *                  index (the skip_bias_row-th (layer, unit) bias row it walks), so the
 *                  epilogue's wait for it runs out and the launch ends with
 *                  KVX_ERR_TIMEOUT in the status word; -1: off.
 * INVALID_ARG for a NULL ctx or values outside those ranges.  Not for production use. */
KVX_API kvx_status kvx_set_test_wait(kvx_ctx* ctx, uint64_t wait_limit_ns, int64_t skip_bias_row);

/* Mapper size in parameters, K plus V (Appendix C, "Serving cost"):
 * CROSS_HEAD 2 L_t n_kv (k n_kv d) d;  PER_HEAD 2 L_t n_kv (k d) d.  -1 on bad input. */
KVX_API int64_t kvx_mapper_params(int32_t tgt_layers, int32_t n_kv_heads, int32_t head_dim, int32_t k,
                          int32_t head_mix);

/* Ridge fit of the per-head mapper on calibration caches (Sec. 3.1, Eq. Wstar; Sec. 3.3
 * for the keys): for every target layer l, K|V and head h, over the N = batch *
 * tokens_per_seq calibration tokens, X = the k selected source layers' head h (keys with
 * the source RoPE stripped) concatenated in selection order, Y = head h of target layer l
 * (keys with the target RoPE stripped), both centred by their column means;
 *   W = (Xc^T Xc + lambda I)^{-1} Xc^T Yc  (lambda on the unnormalised sum),
 *   b = mean(Y) - mean(X) W.
 * `src` holds the source caches [L_s][B][H][T][d] and `tgt` the target caches
 * [L_t][B][H][T][d] of the same tokens (kvx_src layout, bf16, d = 128, 16-byte aligned);
 * `positions` device [batch][tokens_per_seq].  `selection` (host [L_t][k], 1 <= k <= 4)
 * as in kvx_config.  Outputs on the device, fp32: W [L_t][2][H][k*d][d] and
 * b [L_t][2][H][d] (the kvx_config layouts).
 * With head_mix = KVX_CROSS_HEAD the feature is the paper's cross-head concatenation
 * (Sec. 3.1; Appendix "Run information", source-feature row: d_s = k * n_kv * d): X holds
 * every KV head of the k selected layers (layer-major, head-minor) and is shared by all
 * target heads of layer l, so each (l, K|V) is one system (Xc^T Xc + lambda I) W_l =
 * Xc^T Yc_l with F = k*H*128 unknowns and H*128 right-hand sides (Xc^T Xc formed and
 * factored once per target layer, shared across its heads, Sec. 3.1); W is written as
 * [L_t][2][H][k*H*d][d] (k >= 1, k*H*128 <= 16384).  The solve scratch is
 * F*(F + H*128 + 32) float pairs per concurrent system (the matrix, the right-hand sides
 * and the inverted 32 x 32 diagonal blocks of the factor; at most 80 GB, beyond which the
 * systems are factored and solved in waves).  Cross-products of the centred values run
 * on the tensor cores from a bf16 hi + lo split of each value (within 2^-17 of it) and
 * accumulate in fp32; the factorisation and the solves run in float-float arithmetic (each
 * value an unevaluated sum of two fp32 numbers, about 48 significant bits) on the FP32
 * units, the bias too.  Runs on `stream` and
 * synchronises it before returning (an offline step).  Stream-ordered workspace: the
 * blocks (at most L_t*2*H*(k*(k+1)/2 + k)*64 KB), 8 MB per SM, and the packed operands
 * (4 bytes per token, channel, K|V, head and used layer of either model), at most half the
 * free device memory or 32 GB, the tokens taken in chunks beyond that.  INVALID_ARG for
 * bad arguments (a caller workspace that cannot hold 64 tokens included) or when a system
 * is not positive definite (lambda = 0 with too few tokens); DEVICE_BOUNDS when a
 * position is outside [0, 2^24); OOM when the workspace cannot be allocated.  With cfg->workspace the
 * call allocates nothing: the caller's region holds every device piece. */
typedef struct {
  int32_t src_layers, tgt_layers, n_kv_heads, head_dim, k;
  double src_rope_theta, tgt_rope_theta;
  double lambda;                 /* >= 0; the paper's value is 0.01 */
  const int32_t* selection;      /* host [tgt_layers][k], entries in [0, src_layers) */
  void* workspace;               /* device, 256-byte aligned, or NULL (the call allocates) */
  uint64_t workspace_bytes;      /* its size; kvx_fit_workspace_bytes gives the size that
                                  * holds every token in one pass (less: tokens in chunks) */
  const kvx_rope_scaling* src_rope_scaling;   /* NULL: plain theta (see kvx_rope_scaling) */
  const kvx_rope_scaling* tgt_rope_scaling;
  int32_t rope_numerics;        /* kvx_rope_numerics: the strip of both sides' keys */
  int32_t head_mix;             /* kvx_head_mix: KVX_PER_HEAD (0) or KVX_CROSS_HEAD */
} kvx_fit_config;
KVX_API kvx_status kvx_fit_ridge(const kvx_fit_config* cfg, const kvx_src* src, const kvx_src* tgt, int32_t batch,
                                 int32_t tokens_per_seq, const int32_t* positions, float* W, float* b,
                                 void* stream);

/* Workspace bytes for which kvx_fit_ridge (cfg->workspace set) packs every calibration
 * token in one pass; -1 on invalid arguments or when no device is current. */
KVX_API int64_t kvx_fit_workspace_bytes(const kvx_fit_config* cfg, int32_t batch, int32_t tokens_per_seq);

/* Single-source R^2 probe and selection scores (Sec. 2.3, Eq. single_source_ols; Sec.
 * 3.2) on calibration caches: for every target layer l, source layer l', K|V and head h,
 * the OLS fit with intercept of head h of target layer l on head h of source layer l' over
 * the N = batch * tokens_per_seq tokens (keys RoPE-stripped on both sides, theta_s for the
 * source and theta_t for the target), scored by R^2 = 1 - SS_res / SS_tot pooled over
 * the 128 output channels;
 *   scores[l][l'] = (mean_h R^2_K + mean_h R^2_V) / 2,
 * the score that kvx_select_topk / kvx_select_topk_device rank.  `src` [L_s][B][H][T][d]
 * and `tgt` [L_t][B][H][T][d] as in kvx_fit_ridge (bf16, d = 128); `positions` device
 * [batch][tokens_per_seq]; `scores` device double [L_t][L_s]; `r2_kv` device double
 * [2][L_t][L_s] (the head-averaged R^2 of K and of V) or NULL.  The centred
 * cross-products run on the tensor cores as in kvx_fit_ridge (fp32 accumulation of bf16
 * hi + lo products); each source Gram block is factorised in fp64 and inverted, and
 * explained = ||L^{-1} C||^2 is accumulated in fp32.  Runs on `stream` and synchronises
 * it (an offline step).  Workspace: 2 H L_s (L_t + 2) blocks of 64 KB plus the packed
 * operands (as kvx_fit_ridge, every layer of both models); from cfg->workspace when it is
 * set (kvx_r2_probe_workspace_bytes: the size for one pass over the tokens), else
 * stream-ordered allocations.  INVALID_ARG for bad arguments (a caller workspace that
 * cannot hold 64 tokens included), for N <= 128, or when a source Gram block is singular;
 * DEVICE_BOUNDS when a position is outside [0, 2^24); OOM when the workspace cannot be
 * allocated. */
typedef struct {
  int32_t src_layers, tgt_layers, n_kv_heads, head_dim;
  double src_rope_theta, tgt_rope_theta;
  void* workspace;               /* device, 256-byte aligned, or NULL (the call allocates) */
  uint64_t workspace_bytes;
  const kvx_rope_scaling* src_rope_scaling;   /* NULL: plain theta (see kvx_rope_scaling) */
  const kvx_rope_scaling* tgt_rope_scaling;
  int32_t rope_numerics;        /* kvx_rope_numerics: the strip of both sides' keys */
} kvx_probe_config;
KVX_API kvx_status kvx_r2_probe(const kvx_probe_config* cfg, const kvx_src* src, const kvx_src* tgt, int32_t batch,
                                int32_t tokens_per_seq, const int32_t* positions, double* scores, double* r2_kv,
                                void* stream);
KVX_API int64_t kvx_r2_probe_workspace_bytes(const kvx_probe_config* cfg, int32_t batch, int32_t tokens_per_seq);

/* Top-k source-layer selection on the device, with the semantics of kvx_select_topk:
 * `scores` device double [L_t][L_s], `out` device int32 [L_t][k], rows ascending.
 * Synchronises `stream`.  INVALID_ARG for NULL, k outside [1, L_s] or a NaN score. */
KVX_API kvx_status kvx_select_topk_device(const double* scores, int32_t tgt_layers, int32_t src_layers, int32_t k,
                                          int32_t* out, void* stream);

/* MLP mapper apply (Sec. 4.3; Appendix "Run information", MLP baseline architecture):
 * for every target layer l, K|V and head h,
 *   y = W3 relu(W2 relu(W1 x + b1) + b2) + b3
 * (weights in the nn.Linear layout [out][in]) on the cross-head source feature x: the k
 * selected source layers (selection[l], in order) with all H heads each, head-minor,
 * d_s = k H d; keys with the source RoPE stripped and rounded to bf16, values as stored.
 * Keys are re-rotated with the target RoPE after b3.  Accumulation in fp32 on the tensor
 * cores, each hidden activation stored in bf16 after its ReLU, output rounded once to
 * bf16.  bf16 caches and weights, head_dim 128, half-split pairs, hidden a multiple of 256,
 * contiguous targets (UNSUPPORTED for paged).  Weights and biases are DEVICE pointers:
 *   W1 bf16 [L_t][2][H][hidden][d_s]    b1 fp32 [L_t][2][H][hidden]
 *   W2 bf16 [L_t][2][H][hidden][hidden] b2 fp32 [L_t][2][H][hidden]
 *   W3 bf16 [L_t][2][H][d][hidden]      b3 fp32 [L_t][2][H][d]
 * (index 0 of the second axis = K), 16-byte aligned.  Workspace: the stripped source
 * keys and two hidden buffers of 2 B T H hidden bf16 per target layer; from cfg->workspace
 * (kvx_mlp_workspace_bytes: all target layers at once; less processes the target layers
 * in groups) or allocated stream-ordered.  Runs on `stream` and synchronises it, returning
 * the device status (DEVICE_BOUNDS for a position outside [0, 2^24), TIMEOUT if a wait of
 * the kernel ran out).  batch == 0 or tokens_per_seq == 0 is a no-op. */
typedef struct {
  int32_t src_layers, tgt_layers, n_kv_heads, head_dim, k, hidden;
  double src_rope_theta, tgt_rope_theta;
  const int32_t* selection;      /* host [tgt_layers][k], entries in [0, src_layers) */
  const void* W1;
  const float* b1;
  const void* W2;
  const float* b2;
  const void* W3;
  const float* b3;
  void* workspace;               /* device, 256-byte aligned, or NULL (the call allocates) */
  uint64_t workspace_bytes;
  const kvx_rope_scaling* src_rope_scaling;   /* NULL: plain theta (see kvx_rope_scaling) */
  const kvx_rope_scaling* tgt_rope_scaling;
  int32_t rope_numerics;        /* kvx_rope_numerics: source strip and target rotation of keys */
} kvx_mlp_config;
KVX_API kvx_status kvx_mlp_map(const kvx_mlp_config* cfg, const kvx_src* src, int32_t batch, int32_t tokens_per_seq,
                               const int32_t* positions, const kvx_tgt* tgt, void* stream);
KVX_API int64_t kvx_mlp_workspace_bytes(const kvx_mlp_config* cfg, int32_t batch, int32_t tokens_per_seq);

/* Device time in milliseconds of the phases of the last successful kvx_fit_ridge or
 * kvx_r2_probe call on this thread, from CUDA events on the call's stream: ms[0] column
 * sums, ms[1] operand packing, ms[2] tensor-core Gram blocks, ms[3] the solves (fit) or
 * the scores (probe).  `ms` host float[4].  INVALID_ARG if ms is NULL. */
KVX_API kvx_status kvx_last_phase_ms(float* ms);

/* Static description of a status code. */
KVX_API const char* kvx_status_string(kvx_status s);

/* Thread-local description of the last error on this thread ("" if none). */
KVX_API const char* kvx_last_error(void);

/* ---- Mapping with no device allocation (the paper has no counterpart) -------------
 *
 * kvx_create allocates device memory (weight copies, tables, a status word).  Some
 * callers cannot let a library do that: processes whose framework has reserved nearly
 * all device memory for its own pool up front (so a cudaMalloc from a library fails or
 * fragments the pool), and latency-critical serving paths that cannot afford the
 * implicit device synchronisation of cudaMalloc / cudaFree.  kvx_map_noalloc serves them:
 * the caller passes everything in its own buffers (caches, positions, W and bias on the
 * device, the selection table on the host) and the library allocates nothing.  The map
 * runs on the fp32 SIMT kernel, with the same results as kvx_map with KVX_KERNEL_SIMT
 * on a context of the same configuration (rope_numerics included).
 *
 * The little device memory it needs besides the caller's buffers -- a status word and a
 * copy of the selection table -- lives in one fixed array inside libkvx
 * (KVX_NOALLOC_SCRATCH_BYTES, kept by every GPU that loads the library until the process
 * exits).  Consequences:
 *  - The first call on a device looks up that array's device address (cudaGetSymbolAddress,
 *    with the device made current); make that first call before any stream capture.
 *  - Every call on a device shares the array: calls that may overlap on the GPU (other
 *    streams, other host threads) race on it and must be serialised by the caller.  Each
 *    call clears the status word and rewrites the selection copy before its launch.
 *  - tgt_layers * k may not exceed KVX_NOALLOC_MAX_SELECTION (INVALID_ARG otherwise).
 */
#define KVX_NOALLOC_MAX_SELECTION 16384
#define KVX_NOALLOC_SCRATCH_BYTES (256 + 4 * KVX_NOALLOC_MAX_SELECTION)

typedef struct {
  int32_t src_layers, tgt_layers, n_kv_heads, head_dim, k;
  int32_t rope_style;          /* kvx_rope_style */
  double src_rope_theta, tgt_rope_theta;
  int32_t cache_dtype;         /* kvx_dtype of the caches */
  int32_t weight_dtype;        /* kvx_dtype of W */
  int32_t head_mix;            /* kvx_head_mix */
  int32_t reserved;            /* must be 0 */
  const int32_t* selection;    /* HOST [L_t][k], distinct layers in [0, L_s); row block j of W <-> selection[l][j] */
  const void* W;               /* DEVICE [L_t][2][n_kv][F][d] in weight_dtype, 16-byte aligned */
  const float* b;              /* DEVICE fp32 [L_t][2][n_kv][d] (pass zeros for no bias), 16-byte aligned */
  const kvx_rope_scaling* src_rope_scaling;   /* NULL: plain theta */
  const kvx_rope_scaling* tgt_rope_scaling;
  int32_t rope_numerics;       /* kvx_rope_numerics, as in kvx_config (0 = KVX_ROPE_EXACT) */
} kvx_noalloc_mapper;

/* Map as kvx_map does, allocating nothing.  src, tgt, positions, batch and
 * tokens_per_seq are as for kvx_map; `device` is the CUDA device that owns every pointer.
 * Asynchronous on `stream` unless device_status is non-NULL: then the call waits for the
 * stream and stores the device-detected status (KVX_OK, KVX_ERR_DEVICE_BOUNDS) there.
 * Host-detected errors return before any launch, INVALID_ARG among them for a selection
 * row that names a source layer twice.
 *  - The selection table is copied to the device on `stream` (cudaMemcpyAsync): when it
 *    sits in pinned host memory the copy reads it only when the stream reaches it, so
 *    the caller keeps it unchanged until the stream has passed this call.
 *  - Pass device_status = NULL while `stream` is being captured: reading the status waits
 *    for the stream, which a stream under capture does not allow. */
KVX_API kvx_status kvx_map_noalloc(const kvx_noalloc_mapper* m, int device, const kvx_src* src,
                                   int32_t batch, int32_t tokens_per_seq, const int32_t* positions,
                                   const kvx_tgt* tgt, void* stream, int32_t* device_status);

#ifdef __cplusplus
}
#endif

#endif /* KVX_H */
