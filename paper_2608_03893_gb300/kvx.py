"""ctypes binding of the kvx C ABI (include/kvx.h): argument marshalling only.

Each ``kvx_*`` function here calls the C function of the same name in
``lib/libkvx.so`` and raises ``KvxError`` when it returns a status other than
``KVX_OK``.  Every step of the mapping runs in the library's CUDA kernels; nothing in
this module computes any part of it, and there is no fallback: if the shared library
is missing the first call raises.

The ``*_from_tensors`` helpers turn torch tensors (used here only as device memory)
into the plain pointer-and-stride structs of the ABI.
"""
import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "lib", "libkvx.so")

KVX_OK, KVX_ERR_INVALID_ARG, KVX_ERR_UNSUPPORTED, KVX_ERR_OOM = 0, 1, 2, 3
KVX_ERR_CUDA, KVX_ERR_TIMEOUT, KVX_ERR_DEVICE_BOUNDS = 4, 5, 6
KVX_F32, KVX_BF16 = 0, 1
KVX_ROPE_HALF, KVX_ROPE_INTERLEAVED = 0, 1
KVX_ROPE_EXACT, KVX_ROPE_HF = 0, 1
KVX_PER_HEAD, KVX_CROSS_HEAD = 0, 1
KVX_KERNEL_AUTO, KVX_KERNEL_SIMT, KVX_KERNEL_TCGEN05 = 0, 1, 2


class KvxError(RuntimeError):
    def __init__(self, status, where, detail):
        super().__init__("%s: status %d (%s) %s" % (where, status, _status_name(status), detail))
        self.status = status


class kvx_rope_scaling(ctypes.Structure):
    """Llama-3 RoPE frequency scaling (see include/kvx.h)."""
    _fields_ = [("factor", ctypes.c_double), ("low_freq_factor", ctypes.c_double),
                ("high_freq_factor", ctypes.c_double), ("original_max_position", ctypes.c_double)]


_SCALING = [("src_rope_scaling", ctypes.POINTER(kvx_rope_scaling)),
            ("tgt_rope_scaling", ctypes.POINTER(kvx_rope_scaling))]


def rope_scaling(spec):
    """kvx_rope_scaling from (factor, low_freq_factor, high_freq_factor, original_max_position),
    or None."""
    if not spec:
        return None
    return kvx_rope_scaling(*(float(x) for x in spec))


def _scaling_ptr(s):
    return ctypes.pointer(s) if s is not None else ctypes.POINTER(kvx_rope_scaling)()


class kvx_config(ctypes.Structure):
    _fields_ = [
        ("src_layers", ctypes.c_int32), ("tgt_layers", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("k", ctypes.c_int32),
        ("rope_style", ctypes.c_int32), ("src_rope_theta", ctypes.c_double),
        ("tgt_rope_theta", ctypes.c_double), ("cache_dtype", ctypes.c_int32),
        ("weight_dtype", ctypes.c_int32), ("head_mix", ctypes.c_int32), ("reserved", ctypes.c_int32),
        ("selection", ctypes.c_void_p), ("selection_scores", ctypes.c_void_p),
        ("W", ctypes.c_void_p), ("b", ctypes.c_void_p),
    ] + _SCALING + [("rope_numerics", ctypes.c_int32)]


class kvx_src(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("stride", ctypes.c_int64 * 4)]


class kvx_tgt(ctypes.Structure):
    _fields_ = [
        ("paged", ctypes.c_int32), ("block_size", ctypes.c_int32),
        ("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("stride", ctypes.c_int64 * 4),
        ("block_table", ctypes.c_void_p), ("max_blocks_per_seq", ctypes.c_int32),
        ("n_blocks", ctypes.c_int32),
    ]


class kvx_noalloc_mapper(ctypes.Structure):
    _fields_ = [
        ("src_layers", ctypes.c_int32), ("tgt_layers", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("k", ctypes.c_int32),
        ("rope_style", ctypes.c_int32), ("src_rope_theta", ctypes.c_double),
        ("tgt_rope_theta", ctypes.c_double), ("cache_dtype", ctypes.c_int32),
        ("weight_dtype", ctypes.c_int32), ("head_mix", ctypes.c_int32), ("reserved", ctypes.c_int32),
        ("selection", ctypes.c_void_p), ("W", ctypes.c_void_p), ("b", ctypes.c_void_p),
    ] + _SCALING + [("rope_numerics", ctypes.c_int32)]


class kvx_fit_config(ctypes.Structure):
    _fields_ = [
        ("src_layers", ctypes.c_int32), ("tgt_layers", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("k", ctypes.c_int32),
        ("src_rope_theta", ctypes.c_double), ("tgt_rope_theta", ctypes.c_double),
        ("lambda_", ctypes.c_double), ("selection", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_uint64),
    ] + _SCALING + [("rope_numerics", ctypes.c_int32), ("head_mix", ctypes.c_int32)]


class kvx_probe_config(ctypes.Structure):
    _fields_ = [
        ("src_layers", ctypes.c_int32), ("tgt_layers", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("src_rope_theta", ctypes.c_double), ("tgt_rope_theta", ctypes.c_double),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_uint64),
    ] + _SCALING + [("rope_numerics", ctypes.c_int32)]


class kvx_mlp_config(ctypes.Structure):
    _fields_ = [
        ("src_layers", ctypes.c_int32), ("tgt_layers", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("k", ctypes.c_int32),
        ("hidden", ctypes.c_int32),
        ("src_rope_theta", ctypes.c_double), ("tgt_rope_theta", ctypes.c_double),
        ("selection", ctypes.c_void_p),
        ("W1", ctypes.c_void_p), ("b1", ctypes.c_void_p), ("W2", ctypes.c_void_p), ("b2", ctypes.c_void_p),
        ("W3", ctypes.c_void_p), ("b3", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_uint64),
    ] + _SCALING + [("rope_numerics", ctypes.c_int32)]


_lib = None

EXPORTED = ("kvx_create", "kvx_map", "kvx_destroy", "kvx_select_topk", "kvx_get_selection",
            "kvx_set_kernel", "kvx_get_status", "kvx_mapper_params", "kvx_status_string",
            "kvx_last_error", "kvx_map_noalloc", "kvx_fit_ridge", "kvx_last_phase_ms", "kvx_r2_probe",
            "kvx_select_topk_device", "kvx_fit_workspace_bytes", "kvx_r2_probe_workspace_bytes",
            "kvx_mlp_map", "kvx_mlp_workspace_bytes", "kvx_host_pipe_create", "kvx_map_host",
            "kvx_host_pipe_destroy", "kvx_set_test_wait", "kvx_get_kernel", "kvx_tc_load_schedule")


def lib():
    """Load libkvx.so (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("libkvx.so not found at %s: build it with "
                           "`python -m paper_2608_03893_gb300.build`" % LIB_PATH)
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    L.kvx_create.argtypes = [ctypes.POINTER(kvx_config), ctypes.c_int, ctypes.POINTER(vp)]
    L.kvx_map.argtypes = [vp, ctypes.POINTER(kvx_src), i32, i32, vp, ctypes.POINTER(kvx_tgt), vp]
    L.kvx_destroy.argtypes = [vp]
    L.kvx_select_topk.argtypes = [vp, i32, i32, i32, vp]
    L.kvx_get_selection.argtypes = [vp, vp]
    L.kvx_set_kernel.argtypes = [vp, i32]
    L.kvx_get_status.argtypes = [vp, vp]
    L.kvx_mapper_params.argtypes = [i32, i32, i32, i32, i32]
    L.kvx_mapper_params.restype = i64
    L.kvx_status_string.argtypes = [ctypes.c_int]
    L.kvx_status_string.restype = ctypes.c_char_p
    L.kvx_last_error.argtypes = []
    L.kvx_last_error.restype = ctypes.c_char_p
    L.kvx_map_noalloc.argtypes = [ctypes.POINTER(kvx_noalloc_mapper), ctypes.c_int, ctypes.POINTER(kvx_src),
                                  i32, i32, vp, ctypes.POINTER(kvx_tgt), vp, ctypes.POINTER(i32)]
    L.kvx_fit_ridge.argtypes = [ctypes.POINTER(kvx_fit_config), ctypes.POINTER(kvx_src), ctypes.POINTER(kvx_src),
                                i32, i32, vp, vp, vp, vp]
    L.kvx_last_phase_ms.argtypes = [ctypes.POINTER(ctypes.c_float)]
    L.kvx_r2_probe.argtypes = [ctypes.POINTER(kvx_probe_config), ctypes.POINTER(kvx_src), ctypes.POINTER(kvx_src),
                               i32, i32, vp, vp, vp, vp]
    L.kvx_select_topk_device.argtypes = [vp, i32, i32, i32, vp, vp]
    L.kvx_fit_workspace_bytes.argtypes = [ctypes.POINTER(kvx_fit_config), i32, i32]
    L.kvx_fit_workspace_bytes.restype = i64
    L.kvx_r2_probe_workspace_bytes.argtypes = [ctypes.POINTER(kvx_probe_config), i32, i32]
    L.kvx_r2_probe_workspace_bytes.restype = i64
    L.kvx_mlp_map.argtypes = [ctypes.POINTER(kvx_mlp_config), ctypes.POINTER(kvx_src), i32, i32, vp,
                              ctypes.POINTER(kvx_tgt), vp]
    L.kvx_mlp_workspace_bytes.argtypes = [ctypes.POINTER(kvx_mlp_config), i32, i32]
    L.kvx_mlp_workspace_bytes.restype = i64
    L.kvx_host_pipe_create.argtypes = [vp, i32, i32, ctypes.POINTER(vp)]
    L.kvx_map_host.argtypes = [vp, ctypes.POINTER(kvx_src), i32, vp, ctypes.POINTER(kvx_tgt), vp]
    L.kvx_host_pipe_destroy.argtypes = [vp]
    L.kvx_set_test_wait.argtypes = [vp, ctypes.c_uint64, i64]
    L.kvx_get_kernel.argtypes = [vp, i32, ctypes.POINTER(i32)]
    L.kvx_get_kernel.restype = ctypes.c_int
    L.kvx_tc_load_schedule.argtypes = [vp, i32, i32, i32, ctypes.POINTER(i32), vp, vp, vp]
    L.kvx_tc_load_schedule.restype = ctypes.c_int
    L.kvx_set_test_wait.restype = ctypes.c_int
    for name in ("kvx_create", "kvx_map", "kvx_destroy", "kvx_select_topk", "kvx_get_selection",
                 "kvx_set_kernel", "kvx_get_status", "kvx_map_noalloc", "kvx_fit_ridge", "kvx_last_phase_ms",
                 "kvx_r2_probe", "kvx_select_topk_device", "kvx_mlp_map", "kvx_host_pipe_create",
                 "kvx_map_host", "kvx_host_pipe_destroy"):
        getattr(L, name).restype = ctypes.c_int
    _lib = L
    return L


def _status_name(s):
    try:
        return lib().kvx_status_string(s).decode()
    except Exception:
        return str(s)


def _check(status, where):
    if status != KVX_OK:
        raise KvxError(status, where, lib().kvx_last_error().decode())


def _ptr(x):
    """Address of a numpy array or torch tensor (or None)."""
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    return x.ctypes.data


# ------------------------------------------------------------------ ABI calls ----

def kvx_create(cfg, device=0):
    """cfg: kvx_config (host pointers inside must stay alive during the call)."""
    out = ctypes.c_void_p()
    _check(lib().kvx_create(ctypes.byref(cfg), int(device), ctypes.byref(out)), "kvx_create")
    return out


def kvx_map(ctx, src, batch, tokens_per_seq, positions_ptr, tgt, stream=0):
    _check(lib().kvx_map(ctx, ctypes.byref(src), int(batch), int(tokens_per_seq), positions_ptr,
                         ctypes.byref(tgt), stream), "kvx_map")


def kvx_map_noalloc(mapper, device, src, batch, tokens_per_seq, positions_ptr, tgt, stream=0,
                    want_status=True):
    """Map with no allocation by the library (see include/kvx.h).  Returns the device
    status when ``want_status`` (the call then waits for the stream), else None."""
    st = ctypes.c_int32(-1)
    _check(lib().kvx_map_noalloc(ctypes.byref(mapper), int(device), ctypes.byref(src), int(batch),
                                 int(tokens_per_seq), positions_ptr, ctypes.byref(tgt), stream,
                                 ctypes.byref(st) if want_status else None), "kvx_map_noalloc")
    return st.value if want_status else None


KERNEL_NAMES = {1: "simt_map_kernel (fp32 FFMA)", 2: "tc_map_kernel (tcgen05, sm_103a)",
                3: "xh_strip_kernel + tc_xh_kernel (tcgen05 pair GEMM, sm_103a)"}


def kvx_get_kernel(ctx, paged=False):
    """1 SIMT, 2 per-head tensor-core kernel, 3 cross-head tensor-core kernel (see
    include/kvx.h): the kernel kvx_map runs on ctx."""
    out = ctypes.c_int32(0)
    _check(lib().kvx_get_kernel(ctx, int(bool(paged)), ctypes.byref(out)), "kvx_get_kernel")
    return out.value


def kvx_set_test_wait(ctx, wait_limit_ns, skip_bias_row=-1):
    """Test switch of the tensor-core kernel's bounded waits (see include/kvx.h)."""
    _check(lib().kvx_set_test_wait(ctx, int(wait_limit_ns), int(skip_bias_row)), "kvx_set_test_wait")


def kvx_destroy(ctx):
    _check(lib().kvx_destroy(ctx), "kvx_destroy")


def kvx_select_topk(scores, k):
    """scores: float64 numpy [L_t][L_s] (C-contiguous) -> int32 numpy [L_t][k]."""
    import numpy as np
    s = np.ascontiguousarray(scores, dtype=np.float64)
    out = np.empty((s.shape[0], k), dtype=np.int32)
    _check(lib().kvx_select_topk(_ptr(s), s.shape[0], s.shape[1], int(k), _ptr(out)),
           "kvx_select_topk")
    return out


def kvx_tc_load_schedule(selection, src_layers):
    """selection: int32 [L_t][k] -> (load_layer [n_loads], load_word [n_loads], use_word [L_t][k]),
    the per-head tensor-core kernel's source-tile schedule (host only)."""
    import numpy as np
    sel = np.ascontiguousarray(selection, dtype=np.int32)
    Lt, k = sel.shape
    n = ctypes.c_int32(0)
    layer = np.empty(Lt * k, dtype=np.int32)
    word = np.empty(Lt * k, dtype=np.int32)
    use = np.empty((Lt, k), dtype=np.int32)
    _check(lib().kvx_tc_load_schedule(_ptr(sel), int(src_layers), Lt, k, ctypes.byref(n), _ptr(layer), _ptr(word),
                                      _ptr(use)), "kvx_tc_load_schedule")
    return layer[:n.value].copy(), word[:n.value].copy(), use


def kvx_get_selection(ctx, tgt_layers, k):
    import numpy as np
    out = np.empty((tgt_layers, k), dtype=np.int32)
    _check(lib().kvx_get_selection(ctx, _ptr(out)), "kvx_get_selection")
    return out


def kvx_set_kernel(ctx, kernel):
    _check(lib().kvx_set_kernel(ctx, int(kernel)), "kvx_set_kernel")


def kvx_get_status(ctx, stream=0):
    """Returns the device status (int); does not raise for device-detected errors."""
    return lib().kvx_get_status(ctx, stream)


def kvx_mapper_params(tgt_layers, n_kv_heads, head_dim, k, head_mix=KVX_PER_HEAD):
    return lib().kvx_mapper_params(tgt_layers, n_kv_heads, head_dim, k, head_mix)


def kvx_status_string(status):
    return lib().kvx_status_string(int(status)).decode()


def kvx_last_error():
    return lib().kvx_last_error().decode()


# ---------------------------------------------------------- tensor marshalling ----

_DTYPES = {"f32": KVX_F32, "bf16": KVX_BF16}


def dtype_code(t):
    import torch
    if t.dtype == torch.float32:
        return KVX_F32
    if t.dtype == torch.bfloat16:
        return KVX_BF16
    raise TypeError("unsupported dtype %s" % t.dtype)


def config_from_tensors(*, src_layers, tgt_layers, n_kv_heads, head_dim, k, theta_s, theta_t,
                        cache_dtype, W, b=None, selection=None, scores=None,
                        rope_style=KVX_ROPE_HALF, head_mix=KVX_PER_HEAD, rope_scaling=None,
                        rope_numerics=0):
    """Build a kvx_config from host tensors.  Returns (cfg, keepalive) -- hold
    ``keepalive`` until kvx_create returns."""
    import numpy as np
    import torch
    Wc = W.detach().to("cpu").contiguous()
    bc = None if b is None else b.detach().to("cpu").to(Wc.dtype).contiguous()
    sel = None if selection is None else np.ascontiguousarray(selection, dtype=np.int32)
    sc = None if scores is None else np.ascontiguousarray(scores, dtype=np.float64)
    if sel is None and sc is None:
        raise ValueError("need selection or scores")
    cfg = kvx_config()
    cfg.src_layers, cfg.tgt_layers, cfg.n_kv_heads = src_layers, tgt_layers, n_kv_heads
    cfg.head_dim, cfg.k, cfg.rope_style = head_dim, k, rope_style
    cfg.src_rope_theta, cfg.tgt_rope_theta = float(theta_s), float(theta_t)
    cfg.cache_dtype = _DTYPES[cache_dtype] if isinstance(cache_dtype, str) else int(cache_dtype)
    cfg.weight_dtype = dtype_code(Wc)
    cfg.head_mix, cfg.reserved = head_mix, 0
    cfg.selection = _ptr(sel)
    cfg.selection_scores = _ptr(sc)
    cfg.W = _ptr(Wc)
    cfg.b = _ptr(bc)
    rs = globals()["rope_scaling"](rope_scaling)
    cfg.src_rope_scaling = cfg.tgt_rope_scaling = _scaling_ptr(rs)
    cfg.rope_numerics = int(rope_numerics)
    return cfg, (Wc, bc, sel, sc, torch, rs)


def src_from_tensors(k, v):
    """Source caches [L][B][H][T][d] (any strides with d contiguous)."""
    if k.stride() != v.stride() or k.shape != v.shape or k.stride(-1) != 1:
        raise ValueError("source K and V must share shape and strides, head_dim contiguous")
    s = kvx_src()
    s.k, s.v = k.data_ptr(), v.data_ptr()
    for i in range(4):
        s.stride[i] = k.stride(i)
    return s


def tgt_from_tensors(k, v):
    """Contiguous target caches [L][B][H][T][d]."""
    if k.stride() != v.stride() or k.shape != v.shape or k.stride(-1) != 1:
        raise ValueError("target K and V must share shape and strides, head_dim contiguous")
    t = kvx_tgt()
    t.paged, t.block_size = 0, 0
    t.k, t.v = k.data_ptr(), v.data_ptr()
    for i in range(4):
        t.stride[i] = k.stride(i)
    t.block_table, t.max_blocks_per_seq, t.n_blocks = None, 0, 0
    return t


def tgt_paged_from_tensors(k, v, block_table, block_size):
    """Paged target pools [L][n_blocks][H][block_size][d] (strides taken from the
    tensors) and a device int32 block table [B][max_blocks_per_seq]."""
    if k.stride() != v.stride() or k.shape != v.shape or k.stride(-1) != 1:
        raise ValueError("target K and V pools must share shape and strides")
    if k.shape[3] != block_size:
        raise ValueError("pool slot axis must equal block_size")
    t = kvx_tgt()
    t.paged, t.block_size = 1, int(block_size)
    t.k, t.v = k.data_ptr(), v.data_ptr()
    for i in range(4):
        t.stride[i] = k.stride(i)
    t.block_table = block_table.data_ptr()
    t.max_blocks_per_seq = block_table.shape[1]
    t.n_blocks = k.shape[1]
    return t


def _fit_config(src_layers, tgt_layers, n_kv_heads, head_dim, k, theta_s, theta_t, lam, sel, workspace_ptr,
                workspace_bytes, scaling=None):
    cfg = kvx_fit_config(int(src_layers), int(tgt_layers), int(n_kv_heads), int(head_dim), int(k),
                         float(theta_s), float(theta_t), float(lam), _ptr(sel), workspace_ptr,
                         int(workspace_bytes))
    rs = rope_scaling(scaling)
    cfg.src_rope_scaling = cfg.tgt_rope_scaling = _scaling_ptr(rs)
    cfg._rs = rs
    return cfg


def kvx_fit_workspace_bytes(src_layers, tgt_layers, n_kv_heads, head_dim, k, theta_s, theta_t, lam, selection,
                            batch, tokens_per_seq, head_mix=KVX_PER_HEAD):
    """Bytes of a caller workspace that holds every calibration token in one pass (-1 on
    invalid arguments)."""
    import numpy as np
    sel = np.ascontiguousarray(selection, dtype=np.int32)
    cfg = _fit_config(src_layers, tgt_layers, n_kv_heads, head_dim, k, theta_s, theta_t, lam, sel, None, 0)
    cfg.head_mix = int(head_mix)
    return int(lib().kvx_fit_workspace_bytes(ctypes.byref(cfg), int(batch), int(tokens_per_seq)))


def kvx_fit_ridge(src_layers, tgt_layers, n_kv_heads, head_dim, k, theta_s, theta_t, lam, selection,
                  src, tgt, batch, tokens_per_seq, positions_ptr, W_ptr, b_ptr, stream=0,
                  workspace_ptr=None, workspace_bytes=0, rope_scaling=None, rope_numerics=0,
                  head_mix=KVX_PER_HEAD):
    """Ridge fit on calibration caches (see include/kvx.h): src / tgt are kvx_src, selection a
    host int32 [L_t][k] array, W_ptr / b_ptr device fp32 buffers [L_t][2][H][F][d] (F = k*d
    per head, k*H*d cross-head) and [L_t][2][H][d]; an optional caller workspace (device,
    256-byte aligned).  Blocks until the fit is done."""
    import numpy as np
    sel = np.ascontiguousarray(selection, dtype=np.int32)
    cfg = _fit_config(src_layers, tgt_layers, n_kv_heads, head_dim, k, theta_s, theta_t, lam, sel, workspace_ptr,
                      workspace_bytes, rope_scaling)
    cfg.rope_numerics = int(rope_numerics)
    cfg.head_mix = int(head_mix)
    _check(lib().kvx_fit_ridge(ctypes.byref(cfg), ctypes.byref(src), ctypes.byref(tgt), int(batch),
                               int(tokens_per_seq), positions_ptr, W_ptr, b_ptr, stream), "kvx_fit_ridge")


def kvx_last_phase_ms():
    """Device milliseconds of the phases of the last fit / probe call on this thread:
    (column sums, operand packing, tensor-core Gram blocks, solves or scores)."""
    ms = (ctypes.c_float * 4)()
    _check(lib().kvx_last_phase_ms(ms), "kvx_last_phase_ms")
    return tuple(float(x) for x in ms)


def kvx_r2_probe_workspace_bytes(src_layers, tgt_layers, n_kv_heads, head_dim, theta_s, theta_t, batch,
                                 tokens_per_seq):
    """Bytes of a caller workspace for one pass of the probe over the tokens (-1 on invalid
    arguments)."""
    cfg = kvx_probe_config(int(src_layers), int(tgt_layers), int(n_kv_heads), int(head_dim),
                           float(theta_s), float(theta_t), None, 0)
    return int(lib().kvx_r2_probe_workspace_bytes(ctypes.byref(cfg), int(batch), int(tokens_per_seq)))


def kvx_r2_probe(src_layers, tgt_layers, n_kv_heads, head_dim, theta_s, theta_t, src, tgt, batch,
                 tokens_per_seq, positions_ptr, scores_ptr, r2_kv_ptr=None, stream=0,
                 workspace_ptr=None, workspace_bytes=0, rope_scaling=None, rope_numerics=0):
    """Single-source R^2 probe (see include/kvx.h): src / tgt are kvx_src; scores_ptr a
    device float64 [L_t][L_s] buffer, r2_kv_ptr a device float64 [2][L_t][L_s] buffer or
    None; an optional caller workspace.  Blocks until the probe is done."""
    cfg = kvx_probe_config(int(src_layers), int(tgt_layers), int(n_kv_heads), int(head_dim),
                           float(theta_s), float(theta_t), workspace_ptr, int(workspace_bytes))
    rs = globals()["rope_scaling"](rope_scaling)
    cfg.src_rope_scaling = cfg.tgt_rope_scaling = _scaling_ptr(rs)
    cfg.rope_numerics = int(rope_numerics)
    _check(lib().kvx_r2_probe(ctypes.byref(cfg), ctypes.byref(src), ctypes.byref(tgt), int(batch),
                              int(tokens_per_seq), positions_ptr, scores_ptr, r2_kv_ptr, stream),
           "kvx_r2_probe")


def kvx_select_topk_device(scores_ptr, tgt_layers, src_layers, k, out_ptr, stream=0):
    """Top-k selection on the device: scores_ptr device float64 [L_t][L_s], out_ptr device
    int32 [L_t][k] (rows ascending, ties to the lower source index)."""
    _check(lib().kvx_select_topk_device(scores_ptr, int(tgt_layers), int(src_layers), int(k), out_ptr, stream),
           "kvx_select_topk_device")


def mlp_config(src_layers, tgt_layers, n_kv_heads, head_dim, k, hidden, theta_s, theta_t, selection,
               W1_ptr, b1_ptr, W2_ptr, b2_ptr, W3_ptr, b3_ptr, workspace_ptr=None, workspace_bytes=0,
               rope_scaling=None, rope_numerics=0):
    """kvx_mlp_config for kvx_mlp_map (weights and biases DEVICE pointers, see include/kvx.h).
    The returned config keeps the host selection array alive."""
    import numpy as np
    sel = np.ascontiguousarray(selection, dtype=np.int32)
    cfg = kvx_mlp_config(int(src_layers), int(tgt_layers), int(n_kv_heads), int(head_dim), int(k), int(hidden),
                         float(theta_s), float(theta_t), _ptr(sel), W1_ptr, b1_ptr, W2_ptr, b2_ptr, W3_ptr,
                         b3_ptr, workspace_ptr, int(workspace_bytes))
    cfg._sel = sel
    rs = globals()["rope_scaling"](rope_scaling)
    cfg.src_rope_scaling = cfg.tgt_rope_scaling = _scaling_ptr(rs)
    cfg._rs = rs
    cfg.rope_numerics = int(rope_numerics)
    return cfg


def kvx_mlp_workspace_bytes(cfg, batch, tokens_per_seq):
    return int(lib().kvx_mlp_workspace_bytes(ctypes.byref(cfg), int(batch), int(tokens_per_seq)))


def kvx_mlp_map(cfg, src, batch, tokens_per_seq, positions_ptr, tgt, stream=0):
    """MLP mapper apply (see include/kvx.h); blocks until done."""
    _check(lib().kvx_mlp_map(ctypes.byref(cfg), ctypes.byref(src), int(batch), int(tokens_per_seq),
                             positions_ptr, ctypes.byref(tgt), stream), "kvx_mlp_map")


def kvx_host_pipe_create(ctx, batch, chunk_tokens):
    """Staging and streams for kvx_map_host (see include/kvx.h); returns the pipe handle."""
    out = ctypes.c_void_p()
    _check(lib().kvx_host_pipe_create(ctx, int(batch), int(chunk_tokens), ctypes.byref(out)),
           "kvx_host_pipe_create")
    return out.value


def kvx_map_host(pipe, src, tokens_per_seq, positions_ptr, tgt, stream=0):
    """Map host caches (contiguous, ideally pinned) through a pipe; ``stream`` waits for the
    result."""
    _check(lib().kvx_map_host(pipe, ctypes.byref(src), int(tokens_per_seq), positions_ptr, ctypes.byref(tgt),
                              stream), "kvx_map_host")


def kvx_host_pipe_destroy(pipe):
    _check(lib().kvx_host_pipe_destroy(pipe), "kvx_host_pipe_destroy")
