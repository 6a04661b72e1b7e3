"""Python binding of the ResKV C ABI (include/reskv.h).

Argument marshalling only: every step of construction and decode runs in the
CUDA library ``libreskv.so``.  Tensors are passed by ``data_ptr()``; streams
default to torch's current stream.  Importing this module does not load the
library; the first call does, and fails loudly if it has not been built.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libreskv.so")

RESKV_OK = 0
(RESKV_ERR_INVALID_ARG, RESKV_ERR_UNSUPPORTED, RESKV_ERR_OOM, RESKV_ERR_CUDA,
 RESKV_ERR_DEVICE_STATUS) = 1, 2, 3, 4, 5
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "OOM", 4: "CUDA",
                5: "DEVICE_STATUS"}
RESKV_SCORE_OBS_POOL, RESKV_SCORE_KEYNORM = 0, 1
RESKV_GATE_DYNAMIC, RESKV_GATE_FIXED = 0, 1
RESKV_DECODE_AUTO, RESKV_DECODE_FMA, RESKV_DECODE_MMA, RESKV_DECODE_CLUSTER = 0, 1, 2, 3
RESKV_DECODE_LSE_MERGE = 4
RESKV_SOFTMAX_SHARED, RESKV_SOFTMAX_SEPARATE = 0, 1
RESKV_DEBUG_SCORES, RESKV_DEBUG_RANKED, RESKV_DEBUG_LOSSES, RESKV_DEBUG_CANDIDATES = 0, 1, 2, 3
RESKV_DEBUG_UNIT_CANDIDATES = 4
RESKV_BUDGET_UNIFORM, RESKV_BUDGET_ADAKV = 0, 1
RESKV_TEST_FAIL_FIRST_WAIT, RESKV_TEST_FAIL_ALLOC = 1, 2
RESKV_APPEND_FAIL, RESKV_APPEND_RING_DROP, RESKV_APPEND_RING_FOLD = 0, 1, 2
MAX_GRID = 8


class ReskvError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"reskv status {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class reskv_config(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("n_layers", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("group", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("seq_len", ctypes.c_int64),
        ("budget", ctypes.c_int32), ("recent_window", ctypes.c_int32), ("n_obs", ctypes.c_int32),
        ("n_fit", ctypes.c_int32), ("n_val", ctypes.c_int32), ("pool_kernel", ctypes.c_int32),
        ("score_mode", ctypes.c_int32), ("n_grid", ctypes.c_int32),
        ("grid_ratios", ctypes.c_float * MAX_GRID), ("lloyd_iters", ctypes.c_int32),
        ("delta", ctypes.c_float), ("beta", ctypes.c_float),
        ("residual_override", ctypes.POINTER(ctypes.c_int32)),
        ("gate_mode", ctypes.c_int32), ("tau", ctypes.c_float), ("alpha", ctypes.c_float),
        ("g_min", ctypes.c_float), ("g_fixed", ctypes.c_float), ("keep_debug", ctypes.c_int32),
        ("decode_warps", ctypes.c_int32), ("decode_kernel", ctypes.c_int32),
        ("softmax_mode", ctypes.c_int32), ("append_capacity", ctypes.c_int32),
        ("unit_budgets", ctypes.POINTER(ctypes.c_int32)),
        ("budget_mode", ctypes.c_int32), ("adakv_safeguard", ctypes.c_float),
        ("append_policy", ctypes.c_int32),
    ]


class reskv_host_cache(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("n_main", "n_res", "kslots", "vslots", "logc", "slot_pos", "counts", "n_app")]


class reskv_cache_info(ctypes.Structure):
    _fields_ = [("n_units", ctypes.c_int64), ("budget", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("slot_bytes", ctypes.c_int64),
                ("cache_bytes", ctypes.c_int64), ("layer_cluster", ctypes.c_int32),
                ("layer_cluster_warps", ctypes.c_int32), ("all_cluster", ctypes.c_int32),
                ("all_cluster_warps", ctypes.c_int32), ("build_ms", ctypes.c_float * 6),
                ("append_capacity", ctypes.c_int32), ("stride", ctypes.c_int32),
                ("max_appended", ctypes.c_int32), ("ragged", ctypes.c_int32),
                ("total_slots", ctypes.c_int64), ("n_candidates", ctypes.c_int32),
                ("ranked_width", ctypes.c_int32), ("all_units_per_warp", ctypes.c_int32),
                ("layer_units_per_warp", ctypes.c_int32), ("kv_copy_rank", ctypes.c_int32),
                ("reserved0", ctypes.c_int32)]


class reskv_device_cache(ctypes.Structure):
    _fields_ = [("kslots", ctypes.c_void_p), ("vslots", ctypes.c_void_p),
                ("logc", ctypes.c_void_p), ("n_main", ctypes.c_void_p), ("n_res", ctypes.c_void_p),
                ("n_units", ctypes.c_int64), ("budget", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("group", ctypes.c_int32),
                ("gate_mode", ctypes.c_int32), ("tau", ctypes.c_float), ("alpha", ctypes.c_float),
                ("g_min", ctypes.c_float), ("g_fixed", ctypes.c_float)]


_lib = None


def load_library():
    """Load libreskv.so (built in-tree by ``paper_2607_29591_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -m paper_2607_29591_gb300.build` (there is no fallback)")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    cfgp = ctypes.POINTER(reskv_config)
    lib.reskv_config_default.argtypes = [cfgp]
    lib.reskv_config_default.restype = None
    lib.reskv_build_cache.argtypes = [cfgp, ctypes.POINTER(vp), ctypes.POINTER(vp),
                                      ctypes.POINTER(vp), vp, ctypes.POINTER(vp)]
    lib.reskv_build_cache.restype = i32
    lib.reskv_decode_attn.argtypes = [vp, i32, vp, vp, vp]
    lib.reskv_decode_attn.restype = i32
    lib.reskv_decode_attn_layers.argtypes = [vp, i32, i32, vp, vp, vp]
    lib.reskv_decode_attn_layers.restype = i32
    lib.reskv_decode_attn_host.argtypes = [vp, vp, vp, vp]
    lib.reskv_decode_attn_host.restype = i32
    lib.reskv_free.argtypes = [vp]
    lib.reskv_free.restype = None
    lib.reskv_last_error.argtypes = []
    lib.reskv_last_error.restype = ctypes.c_char_p
    lib.reskv_check_status.argtypes = [vp]
    lib.reskv_check_status.restype = i32
    lib.reskv_get_info.argtypes = [vp, ctypes.POINTER(reskv_cache_info)]
    lib.reskv_get_info.restype = i32
    lib.reskv_get_unit_budgets.argtypes = [vp, ctypes.POINTER(ctypes.c_int32), ctypes.c_int64]
    lib.reskv_get_unit_budgets.restype = i32
    lib.reskv_import_cache.argtypes = [cfgp, ctypes.POINTER(reskv_host_cache), vp,
                                       ctypes.POINTER(vp)]
    lib.reskv_import_cache.restype = i32
    lib.reskv_export_cache.argtypes = [vp, ctypes.POINTER(reskv_host_cache), vp]
    lib.reskv_export_cache.restype = i32
    lib.reskv_export_debug.argtypes = [vp, i32, vp, sz]
    lib.reskv_export_debug.restype = i32
    lib.reskv_append.argtypes = [vp, i32, vp, vp, vp]
    lib.reskv_append.restype = i32
    lib.reskv_decode_attn_noalloc.argtypes = [ctypes.POINTER(reskv_device_cache), vp, vp, vp]
    lib.reskv_decode_attn_noalloc.restype = i32
    lib.reskv_noalloc_check_status.argtypes = [vp, ctypes.POINTER(ctypes.c_int32)]
    lib.reskv_noalloc_check_status.restype = i32
    lib.reskv_test_inject.argtypes = [i32, ctypes.c_int64]
    lib.reskv_test_inject.restype = i32
    _lib = lib
    return lib


def _check(status: int):
    if status != RESKV_OK:
        raise ReskvError(status, load_library().reskv_last_error().decode())


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _dptr(t, dtype_name: str, what: str):
    """Device pointer of a contiguous CUDA tensor of the expected dtype."""
    if not t.is_cuda:
        raise ValueError(f"{what} must be a CUDA tensor")
    if str(t.dtype) != dtype_name:
        raise ValueError(f"{what} must be {dtype_name}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


class Cache:
    """Owning wrapper of a reskv_cache* handle (freed with reskv_free)."""

    def __init__(self, handle: ctypes.c_void_p, cfg: reskv_config):
        self.handle = handle
        self.cfg = cfg

    def free(self):
        if self.handle:
            load_library().reskv_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def reskv_config_default(**fields) -> reskv_config:
    """reskv_config with the paper's defaults, then ``fields`` applied.

    ``grid_ratios`` may be a sequence (sets n_grid); ``residual_override`` and
    ``unit_budgets`` numpy int32 arrays per unit (kept alive on the returned
    struct).
    """
    cfg = reskv_config()
    load_library().reskv_config_default(ctypes.byref(cfg))
    for k, v in fields.items():
        if k == "grid_ratios":
            vals = list(v)
            cfg.n_grid = len(vals)
            for i in range(MAX_GRID):
                cfg.grid_ratios[i] = vals[i] if i < len(vals) else 0.0
        elif k in ("residual_override", "unit_budgets"):
            if v is None:
                setattr(cfg, k, None)
                setattr(cfg, f"_{k}_keepalive", None)
            else:
                arr = np.ascontiguousarray(v, dtype=np.int32)
                setattr(cfg, f"_{k}_keepalive", arr)
                setattr(cfg, k, arr.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
        else:
            setattr(cfg, k, v)
    return cfg


def reskv_last_error() -> str:
    return load_library().reskv_last_error().decode()


def reskv_build_cache(cfg: reskv_config, K_layers: Sequence, V_layers: Sequence,
                      Qobs_layers: Optional[Sequence] = None, stream=None) -> Cache:
    """Alg. 1 on the GPU.  K_layers[l], V_layers[l]: bf16 [B, H_kv, s, d] CUDA
    tensors; Qobs_layers[l]: bf16 [B, H_kv*G, n_obs, d] or None."""
    L = cfg.n_layers
    if len(K_layers) != L or len(V_layers) != L:
        raise ValueError("one K and one V tensor per layer")
    kp = (ctypes.c_void_p * L)(*[_dptr(k, "torch.bfloat16", "K").value for k in K_layers])
    vp = (ctypes.c_void_p * L)(*[_dptr(v, "torch.bfloat16", "V").value for v in V_layers])
    qp = None
    if Qobs_layers is not None:
        if len(Qobs_layers) != L:
            raise ValueError("one Qobs tensor per layer")
        qp = (ctypes.c_void_p * L)(*[_dptr(q, "torch.bfloat16", "Qobs").value
                                     for q in Qobs_layers])
    out = ctypes.c_void_p()
    _check(load_library().reskv_build_cache(ctypes.byref(cfg), kp, vp, qp, _stream(stream),
                                            ctypes.byref(out)))
    return Cache(out, cfg)


def reskv_decode_attn(cache: Cache, layer: int, Q, O, stream=None) -> None:
    """Alg. 2.  layer >= 0: Q bf16 [B, H_q, d], O fp32 [B, H_q, d]; layer == -1:
    every layer, Q [L, B, H_q, d] and O likewise."""
    c = cache.cfg
    need = (c.n_layers if layer == -1 else 1) * c.batch * c.n_kv_heads * c.group * c.head_dim
    for name, t in (("Q", Q), ("O", O)):
        if t.numel() != need:
            raise ValueError(f"{name} holds {t.numel()} elements; this call needs {need}")
    _check(load_library().reskv_decode_attn(cache.handle, int(layer),
                                            _dptr(Q, "torch.bfloat16", "Q"),
                                            _dptr(O, "torch.float32", "O"), _stream(stream)))


def reskv_decode_attn_layers(cache: Cache, layer0: int, n_layers: int, Q, O, stream=None) -> None:
    """Alg. 2 for layers layer0 .. layer0 + n_layers - 1 in one launch: Q bf16
    [n_layers, B, H_q, d], O fp32 likewise."""
    c = cache.cfg
    need = int(n_layers) * c.batch * c.n_kv_heads * c.group * c.head_dim
    for name, t in (("Q", Q), ("O", O)):
        if t.numel() != need:
            raise ValueError(f"{name} holds {t.numel()} elements; this call needs {need}")
    _check(load_library().reskv_decode_attn_layers(cache.handle, int(layer0), int(n_layers),
                                                   _dptr(Q, "torch.bfloat16", "Q"),
                                                   _dptr(O, "torch.float32", "O"),
                                                   _stream(stream)))


def _hptr(t, dtype_name: str, what: str):
    """Host pointer of a contiguous CPU tensor of the expected dtype."""
    if t.is_cuda:
        raise ValueError(f"{what} must be a host (CPU) tensor")
    if str(t.dtype) != dtype_name:
        raise ValueError(f"{what} must be {dtype_name}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def reskv_decode_attn_host(cache: Cache, Q_host, O_host, stream=None) -> None:
    """Alg. 2 for every layer with host buffers (pinned for overlap): Q_host
    bf16 [L, B, H_q, d], O_host fp32 likewise.  Asynchronous: O_host is
    complete once the stream has passed the call."""
    c = cache.cfg
    need = c.n_layers * c.batch * c.n_kv_heads * c.group * c.head_dim
    for name, t in (("Q_host", Q_host), ("O_host", O_host)):
        if t.numel() != need:
            raise ValueError(f"{name} holds {t.numel()} elements; this call needs {need}")
    _check(load_library().reskv_decode_attn_host(cache.handle,
                                                 _hptr(Q_host, "torch.bfloat16", "Q_host"),
                                                 _hptr(O_host, "torch.float32", "O_host"),
                                                 _stream(stream)))


def reskv_append(cache: Cache, layer: int, K_new, V_new, stream=None) -> None:
    """Append one token per (batch, KV head) unit: layer >= 0: K_new, V_new
    bf16 [B, H_kv, d]; layer == -1: [L, B, H_kv, d]."""
    c = cache.cfg
    need = (c.n_layers if layer == -1 else 1) * c.batch * c.n_kv_heads * c.head_dim
    for name, t in (("K_new", K_new), ("V_new", V_new)):
        if t.numel() != need:
            raise ValueError(f"{name} holds {t.numel()} elements; this call needs {need}")
    _check(load_library().reskv_append(cache.handle, int(layer),
                                       _dptr(K_new, "torch.bfloat16", "K_new"),
                                       _dptr(V_new, "torch.bfloat16", "V_new"), _stream(stream)))


def reskv_test_inject(what: int, n: int) -> None:
    """Testing only: inject a decode wait timeout or an allocation failure
    (see include/reskv.h)."""
    _check(load_library().reskv_test_inject(int(what), int(n)))


def reskv_free(cache: Cache) -> None:
    cache.free()


def reskv_check_status(cache: Cache) -> None:
    _check(load_library().reskv_check_status(cache.handle))


def reskv_get_info(cache: Cache) -> dict:
    info = reskv_cache_info()
    _check(load_library().reskv_get_info(cache.handle, ctypes.byref(info)))
    out = {f: getattr(info, f) for f, _ in info._fields_}
    out["build_ms"] = list(out["build_ms"])
    return out


def reskv_get_unit_budgets(cache: Cache) -> np.ndarray:
    """Budget b_u of every unit of the handle's layout: int32 [U]."""
    c = cache.cfg
    U = c.n_layers * c.batch * c.n_kv_heads
    out = np.zeros(U, np.int32)
    _check(load_library().reskv_get_unit_budgets(
        cache.handle, out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), U))
    return out


def _host_view(arrs: dict) -> reskv_host_cache:
    h = reskv_host_cache()
    for k, _ in h._fields_:
        a = arrs.get(k)
        setattr(h, k, None if a is None else a.ctypes.data)
    return h


def reskv_import_cache(cfg: reskv_config, n_main, n_res, kslots, vslots, logc,
                       slot_pos=None, counts=None, n_app=None, stream=None) -> Cache:
    """Build a handle from host numpy arrays (layout as in include/reskv.h):
    kslots/vslots uint16 bf16 bits [U, S, d], logc float32 [U, S], with the
    unit stride S = budget + append_capacity."""
    arrs = dict(n_main=np.ascontiguousarray(n_main, np.int32),
                n_res=np.ascontiguousarray(n_res, np.int32),
                kslots=np.ascontiguousarray(kslots, np.uint16),
                vslots=np.ascontiguousarray(vslots, np.uint16),
                logc=np.ascontiguousarray(logc, np.float32),
                slot_pos=None if slot_pos is None else np.ascontiguousarray(slot_pos, np.int32),
                counts=None if counts is None else np.ascontiguousarray(counts, np.int32),
                n_app=None if n_app is None else np.ascontiguousarray(n_app, np.int32))
    U, d = cfg.n_layers * cfg.batch * cfg.n_kv_heads, cfg.head_dim
    N = unit_offsets(cfg)[-1]
    for k in ("kslots", "vslots", "logc", "slot_pos", "counts"):
        if arrs[k] is not None:                  # [U, S, ...] or flat [N, ...]
            arrs[k] = arrs[k].reshape((N, d) if k in ("kslots", "vslots") else (N,))
    for k, shape in (("n_main", (U,)), ("n_res", (U,)), ("kslots", (N, d)),
                     ("vslots", (N, d)), ("logc", (N,)), ("slot_pos", (N,)),
                     ("counts", (N,)), ("n_app", (U,))):
        if arrs[k] is not None and arrs[k].shape != shape:
            raise ValueError(f"{k} must have shape {shape}, got {arrs[k].shape}")
    h = _host_view(arrs)
    out = ctypes.c_void_p()
    _check(load_library().reskv_import_cache(ctypes.byref(cfg), ctypes.byref(h), _stream(stream),
                                             ctypes.byref(out)))
    return Cache(out, cfg)


def reskv_export_cache(cache: Cache, stream=None) -> dict:
    """Copy the cache layout to host numpy arrays."""
    cfg = cache.cfg
    U, d = cfg.n_layers * cfg.batch * cfg.n_kv_heads, cfg.head_dim
    ragged = bool(reskv_get_info(cache)["ragged"])
    off = (np.concatenate([[0], np.cumsum(reskv_get_unit_budgets(cache).astype(np.int64)
                                          + cfg.append_capacity)])
           if ragged else unit_offsets(cfg))
    N = off[-1]
    arrs = dict(n_main=np.zeros(U, np.int32), n_res=np.zeros(U, np.int32),
                kslots=np.zeros((N, d), np.uint16), vslots=np.zeros((N, d), np.uint16),
                logc=np.zeros(N, np.float32), slot_pos=np.zeros(N, np.int32),
                counts=np.zeros(N, np.int32), n_app=np.zeros(U, np.int32))
    h = _host_view(arrs)
    _check(load_library().reskv_export_cache(cache.handle, ctypes.byref(h), _stream(stream)))
    if ragged:                                   # per-unit budgets: flat arrays plus offsets
        arrs["offsets"] = off
    else:                                        # one stride: [U, S, ...]
        S = cfg.budget + cfg.append_capacity
        for k in ("kslots", "vslots"):
            arrs[k] = arrs[k].reshape(U, S, d)
        for k in ("logc", "slot_pos", "counts"):
            arrs[k] = arrs[k].reshape(U, S)
    return arrs


def unit_offsets(cfg: reskv_config) -> np.ndarray:
    """First slot of every unit (and the total) for cfg's layout: [U + 1]."""
    U = cfg.n_layers * cfg.batch * cfg.n_kv_heads
    if cfg.unit_budgets:
        sizes = np.ctypeslib.as_array(cfg.unit_budgets, shape=(U,)).astype(np.int64)
    else:
        sizes = np.full(U, cfg.budget, np.int64)
    return np.concatenate([[0], np.cumsum(sizes + cfg.append_capacity)]).astype(np.int64)


def reskv_export_debug(cache: Cache, what: int, n_cand: Optional[int] = None) -> np.ndarray:
    """Construction intermediates (cfg.keep_debug must have been set, except
    for the candidate tables).  ``n_cand`` defaults to the handle's count."""
    cfg = cache.cfg
    U = cfg.n_layers * cfg.batch * cfg.n_kv_heads
    s = cfg.seq_len
    info = reskv_get_info(cache)
    nc = info["n_candidates"] if n_cand is None else n_cand
    if what == RESKV_DEBUG_CANDIDATES:
        out = np.zeros(nc, np.int32)
    elif what == RESKV_DEBUG_UNIT_CANDIDATES:
        out = np.zeros((U, nc), np.int32)
    elif what == RESKV_DEBUG_SCORES:
        out = np.zeros((U, s), np.float64)
    elif what == RESKV_DEBUG_RANKED:
        out = np.zeros((U, info["ranked_width"]), np.int32)
    elif what == RESKV_DEBUG_LOSSES:
        out = np.zeros((U, 1 + nc), np.float64)
    else:
        raise ValueError("unknown debug array")
    _check(load_library().reskv_export_debug(cache.handle, int(what),
                                             ctypes.c_void_p(out.ctypes.data), out.nbytes))
    return out


def reskv_decode_attn_noalloc(kslots, vslots, logc, n_main, n_res, n_kv_heads: int, group: int,
                              Q, O, gate_mode: int = RESKV_GATE_DYNAMIC, tau: float = 0.25,
                              alpha: float = 12.0, g_min: float = 0.0, g_fixed: float = 1.0,
                              stream=None) -> None:
    """Decode from a cache held in the caller's own device tensors, with no
    device allocation by the library (see include/reskv.h).

    kslots, vslots: bf16 [U, b, 128]; logc: float32 [U, b]; n_main, n_res:
    int32 [U]; Q: bf16 [U / n_kv_heads, n_kv_heads * group, 128]; O: float32,
    Q's shape.  Every shape is checked here, before the call: the kernel reads
    and writes inside these arrays by their sizes alone.
    """
    if kslots.dim() != 3 or int(kslots.shape[2]) != 128:
        raise ValueError(f"kslots must be [U, b, 128], got {tuple(kslots.shape)}")
    U, b = int(kslots.shape[0]), int(kslots.shape[1])
    H, G = int(n_kv_heads), int(group)
    if H < 1 or U % H != 0:
        raise ValueError(f"n_units {U} is not a multiple of n_kv_heads {H}")
    # row-major arrays of these many elements (any leading shape)
    for name, t, n in (("vslots", vslots, U * b * 128), ("logc", logc, U * b),
                       ("n_main", n_main, U), ("n_res", n_res, U),
                       ("Q", Q, U * G * 128), ("O", O, U * G * 128)):
        if t.numel() != n or (name in ("vslots", "Q", "O") and int(t.shape[-1]) != 128):
            raise ValueError(f"{name} must hold {n} elements (rows of 128 for vslots, Q, O), "
                             f"got shape {tuple(t.shape)}")
    d = reskv_device_cache(
        kslots=_dptr(kslots, "torch.bfloat16", "kslots").value,
        vslots=_dptr(vslots, "torch.bfloat16", "vslots").value,
        logc=_dptr(logc, "torch.float32", "logc").value,
        n_main=_dptr(n_main, "torch.int32", "n_main").value,
        n_res=_dptr(n_res, "torch.int32", "n_res").value,
        n_units=U, budget=b, n_kv_heads=H, group=G,
        gate_mode=int(gate_mode), tau=tau, alpha=alpha, g_min=g_min, g_fixed=g_fixed)
    _check(load_library().reskv_decode_attn_noalloc(ctypes.byref(d),
                                                    _dptr(Q, "torch.bfloat16", "Q"),
                                                    _dptr(O, "torch.float32", "O"),
                                                    _stream(stream)))


def reskv_noalloc_check_status(stream=None) -> int:
    """Read and clear the no-allocation decode's device status word; raises
    ReskvError (RESKV_ERR_DEVICE_STATUS) if a kernel fault was recorded.
    Returns the kernel the thread's last call launched (RESKV_DECODE_MMA or
    RESKV_DECODE_FMA, 0 before the first call)."""
    k = ctypes.c_int32(0)
    _check(load_library().reskv_noalloc_check_status(_stream(stream), ctypes.byref(k)))
    return int(k.value)
