"""Thin Python binding of libswan (ctypes).  Argument marshalling only: every
step of the decode path runs in the library's CUDA kernels.  PyTorch supplies
device memory and the stream.

The library must have been built (``paper_2511_18936_gb300.build.build()``);
loading fails loudly otherwise - there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libswan.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CAPACITY, ERR_CUDA, ERR_STATE, \
    ERR_DEVICE_TIMEOUT, ERR_NOMEM, ERR_DEVICE_CHECK = range(9)
EXPORT_BUFFER_K, EXPORT_BUFFER_V, EXPORT_SPARSE_K, EXPORT_SPARSE_V = 1, 2, 3, 4
VALUE_FORMATS = {"fp16": 0, "fp8_e4m3": 1}
KERNEL_ROTATE_Q, KERNEL_DECODE, KERNEL_COMBINE, KERNEL_APPEND, KERNEL_PRUNE = range(5)
KERNEL_KINDS = 8
FAULT_ALLOC, FAULT_LAUNCH = 1, 2
KERNEL_NAMES = {KERNEL_ROTATE_Q: "rotate_q", KERNEL_DECODE: "decode", KERNEL_COMBINE: "combine",
                KERNEL_APPEND: "append", KERNEL_PRUNE: "prune_ring"}

# Every symbol include/swan.h and include/swan_basis.h declare.
EXPORTED = ["swan_init", "swan_destroy", "swan_set_k", "swan_append", "swan_flush_buffer",
            "swan_decode", "swan_query", "swan_debug_export", "swan_check",
            "swan_timing_enable", "swan_timing_read", "swan_launch_count",
            "swan_status_string", "swan_last_error", "swan_decode_noalloc", "swan_set_kv",
            "swan_gram_workspace_bytes", "swan_gram", "swan_basis_eig", "swan_energy",
            "swan_basis_check", "swan_append_varlen", "swan_reset_sequence", "swan_fork_sequence",
            "swan_query_lengths", "swan_debug_export_seq", "swan_append_decode", "swan_debug_fail_after",
            "swan_debug_check_guards", "swan_noalloc_check", "swan_debug_starve_tc"]


class SwanConfig(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int), ("batch", ctypes.c_int),
                ("n_q_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("k_store", ctypes.c_int),
                ("buffer_cap", ctypes.c_int), ("max_seq", ctypes.c_int),
                ("page_tokens", ctypes.c_int), ("stream", ctypes.c_void_p),
                ("value_format", ctypes.c_int), ("k_store_v", ctypes.c_int), ("pool_pages", ctypes.c_int)]


class LayerInfo(ctypes.Structure):
    _fields_ = [("sparse_len", ctypes.c_int64), ("buffer_len", ctypes.c_int64),
                ("k_active", ctypes.c_int), ("k_store", ctypes.c_int), ("k_slots", ctypes.c_int),
                ("page_tokens", ctypes.c_int), ("page_bytes", ctypes.c_int64),
                ("device_bytes", ctypes.c_int64), ("value_format", ctypes.c_int),
                ("k_active_v", ctypes.c_int), ("k_store_v", ctypes.c_int), ("k_slots_v", ctypes.c_int),
                ("uniform", ctypes.c_int), ("pool_pages", ctypes.c_int64), ("free_pages", ctypes.c_int64)]


class Timing(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_double * KERNEL_KINDS), ("launches", ctypes.c_int64 * KERNEL_KINDS)]


class CacheView(ctypes.Structure):
    """A cache in caller-owned device memory (see swan_decode_noalloc)."""
    _fields_ = [("pages", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
                ("num_pages", ctypes.c_int64), ("pages_per_unit", ctypes.c_int),
                ("page_tokens", ctypes.c_int), ("k_slots", ctypes.c_int), ("k_active", ctypes.c_int),
                ("buf_k", ctypes.c_void_p), ("buf_v", ctypes.c_void_p), ("buffer_cap", ctypes.c_int),
                ("buf_start", ctypes.c_int), ("buf_len", ctypes.c_int), ("sparse_len", ctypes.c_int64),
                ("batch", ctypes.c_int), ("n_q_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("R_qk", ctypes.c_void_p), ("R_vo_t", ctypes.c_void_p),
                ("value_format", ctypes.c_int), ("k_slots_v", ctypes.c_int), ("k_active_v", ctypes.c_int)]


class SwanVectors(ctypes.Structure):
    """A set of fp16 vectors in device memory (see swan_basis.h)."""
    _fields_ = [("data", ctypes.c_void_p), ("n_mats", ctypes.c_int), ("group", ctypes.c_int),
                ("count", ctypes.c_int64), ("stride_mat", ctypes.c_int64),
                ("stride_group", ctypes.c_int64), ("stride_pos", ctypes.c_int64),
                ("stride_coord", ctypes.c_int64)]


class SwanError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: status {status} ({detail})")
        self.status = status


_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libswan.so (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with "
                           "`python -m paper_2511_18936_gb300.build` (no fallback exists)")
    lib = ctypes.CDLL(path)
    vp, i, i64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64
    sig = {
        "swan_init": (i, [ctypes.POINTER(vp), ctypes.POINTER(SwanConfig), vp, vp]),
        "swan_destroy": (i, [vp]),
        "swan_set_k": (i, [vp, i]),
        "swan_set_kv": (i, [vp, i, i]),
        "swan_append": (i, [vp, i, vp, vp, i]),
        "swan_append_varlen": (i, [vp, i, vp, vp, i, ctypes.POINTER(ctypes.c_int32)]),
        "swan_reset_sequence": (i, [vp, i]),
        "swan_fork_sequence": (i, [vp, i, i]),
        "swan_query_lengths": (i, [vp, i, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int32)]),
        "swan_debug_export_seq": (i, [vp, i, i, i, vp, ctypes.c_size_t]),
        "swan_flush_buffer": (i, [vp, i]),
        "swan_decode": (i, [vp, i, vp, vp]),
        "swan_append_decode": (i, [vp, i, vp, vp, i, ctypes.POINTER(ctypes.c_int32), vp, vp]),
        "swan_query": (i, [vp, i, ctypes.POINTER(LayerInfo)]),
        "swan_debug_export": (i, [vp, i, i, vp, ctypes.c_size_t]),
        "swan_check": (i, [vp]),
        "swan_timing_enable": (i, [vp, i]),
        "swan_timing_read": (i, [vp, ctypes.POINTER(Timing)]),
        "swan_launch_count": (i64, [vp]),
        "swan_status_string": (ctypes.c_char_p, [i]),
        "swan_last_error": (ctypes.c_char_p, []),
        "swan_decode_noalloc": (i, [ctypes.POINTER(CacheView), vp, vp, vp]),
        "swan_noalloc_check": (i, [vp]),
        "swan_debug_starve_tc": (i, [i64]),
        "swan_gram_workspace_bytes": (ctypes.c_size_t, [i]),
        "swan_gram": (i, [ctypes.POINTER(SwanVectors), vp, i, vp, ctypes.c_size_t, vp]),
        "swan_basis_eig": (i, [vp, i, vp, vp, vp, vp]),
        "swan_energy": (i, [ctypes.POINTER(SwanVectors), vp, vp, i, vp]),
        "swan_basis_check": (i, [vp, vp]),
        "swan_debug_fail_after": (i, [i, i64]),
        "swan_debug_check_guards": (i, [vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(status: int, where: str):
    if status != OK:
        lib = load_library()
        detail = lib.swan_last_error().decode() or lib.swan_status_string(status).decode()
        raise SwanError(status, where, detail)


def _ptr(t) -> int:
    """Device address of a contiguous CUDA tensor (or a raw int address)."""
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("tensor must live on the GPU")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


class Context:
    """One SWAN cache (``num_layers`` layers) on the current CUDA device.

    ``R_qk``/``R_vo``: CUDA fp32 tensors ``[num_layers][n_kv_heads][128][128]``.
    ``stream``: a ``torch.cuda.Stream`` (default: the current stream).
    """

    def __init__(self, R_qk, R_vo=None, *, num_layers: int, batch: int, n_q_heads: int,
                 n_kv_heads: int, k_store: int, buffer_cap: int, max_seq: int,
                 page_tokens: int = 0, head_dim: int = 128, stream=None,
                 value_format: str = "fp16", k_store_v: int = 0, pool_pages: int = 0):
        import torch
        self._lib = load_library()
        if stream is None:
            stream = torch.cuda.current_stream()
        self.stream = stream
        if value_format not in VALUE_FORMATS:
            raise ValueError(f"value_format must be one of {sorted(VALUE_FORMATS)}")
        self.cfg = SwanConfig(num_layers, batch, n_q_heads, n_kv_heads, head_dim, k_store,
                              buffer_cap, max_seq, page_tokens, ctypes.c_void_p(stream.cuda_stream),
                              VALUE_FORMATS[value_format], k_store_v, pool_pages)
        self.batch, self.n_q_heads, self.n_kv_heads = batch, n_q_heads, n_kv_heads
        self.num_layers, self.k_store, self.head_dim = num_layers, k_store, head_dim
        self.k_store_v = k_store_v or k_store
        h = ctypes.c_void_p()
        _check(self._lib.swan_init(ctypes.byref(h), ctypes.byref(self.cfg), _ptr(R_qk),
                                   None if R_vo is None else _ptr(R_vo)), "swan_init")
        self._h = h

    # -- lifecycle ----------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None):
            self._lib.swan_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- the hot path ------------------------------------------------------
    def set_k(self, k_active: int, k_active_v: int | None = None):
        if k_active_v is None:
            _check(self._lib.swan_set_k(self._h, int(k_active)), "swan_set_k")
        else:
            _check(self._lib.swan_set_kv(self._h, int(k_active), int(k_active_v)), "swan_set_kv")

    def append(self, layer: int, k_new, v_new, T: int | None = None, n_new=None):
        """Append ``T`` tokens per row (``k_new``/``v_new`` ``[B][H][T][d]``), or
        ``n_new[b]`` of them to row b (a host sequence of ``batch`` ints)."""
        if T is None:
            T = k_new.shape[2]
        if n_new is None:
            _check(self._lib.swan_append(self._h, int(layer), _ptr(k_new), _ptr(v_new), int(T)),
                   "swan_append")
            return
        counts = (ctypes.c_int32 * self.batch)(*[int(x) for x in n_new])
        _check(self._lib.swan_append_varlen(self._h, int(layer), _ptr(k_new), _ptr(v_new), int(T), counts),
               "swan_append_varlen")

    def reset_sequence(self, b: int):
        _check(self._lib.swan_reset_sequence(self._h, int(b)), "swan_reset_sequence")

    def fork_sequence(self, src: int, dst: int):
        """Row dst becomes a copy of row src (shared pages, copied buffer)."""
        _check(self._lib.swan_fork_sequence(self._h, int(src), int(dst)), "swan_fork_sequence")

    def lengths(self, layer: int = 0):
        """Per-row (sparse, buffered) token counts of a layer."""
        sp = (ctypes.c_int64 * self.batch)()
        bf = (ctypes.c_int32 * self.batch)()
        _check(self._lib.swan_query_lengths(self._h, int(layer), sp, bf), "swan_query_lengths")
        return list(sp), list(bf)

    def flush(self, layer: int = -1):
        _check(self._lib.swan_flush_buffer(self._h, int(layer)), "swan_flush_buffer")

    def decode(self, layer: int, q, out=None):
        if out is None:
            import torch
            out = torch.empty_like(q)
        _check(self._lib.swan_decode(self._h, int(layer), _ptr(q), _ptr(out)), "swan_decode")
        return out

    def append_decode(self, layer: int, k_new, v_new, q, out=None, T: int | None = None, n_new=None):
        """One serving step: ``append(layer, k_new, v_new, T, n_new)`` then
        ``decode(layer, q, out)`` (the query rotation runs inside the append's
        launch for a decode-step append)."""
        if T is None:
            T = k_new.shape[2]
        if out is None:
            import torch
            out = torch.empty_like(q)
        counts = None if n_new is None else (ctypes.c_int32 * self.batch)(*[int(x) for x in n_new])
        _check(self._lib.swan_append_decode(self._h, int(layer), _ptr(k_new), _ptr(v_new), int(T), counts,
                                            _ptr(q), _ptr(out)), "swan_append_decode")
        return out

    # -- inspection --------------------------------------------------------
    def query(self, layer: int = 0) -> LayerInfo:
        info = LayerInfo()
        _check(self._lib.swan_query(self._h, int(layer), ctypes.byref(info)), "swan_query")
        return info

    def check(self):
        _check(self._lib.swan_check(self._h), "swan_check")

    def check_guards(self):
        """Raise if a kernel wrote into the guard regions around any device buffer."""
        _check(self._lib.swan_debug_check_guards(self._h), "swan_debug_check_guards")

    def export_buffer(self, layer: int, which: str) -> np.ndarray:
        info = self.query(layer)
        shape = (self.batch, self.n_kv_heads, info.buffer_len, self.head_dim)
        out = np.empty(shape, np.float16)
        what = EXPORT_BUFFER_K if which == "k" else EXPORT_BUFFER_V
        _check(self._lib.swan_debug_export(self._h, int(layer), what,
                                           out.ctypes.data_as(ctypes.c_void_p), out.nbytes),
               "swan_debug_export")
        return out

    def export_sparse(self, layer: int, which: str):
        info = self.query(layer)
        shape = (self.batch, self.n_kv_heads, info.sparse_len,
                 self.k_store if which == "k" else self.k_store_v)
        n = int(np.prod(shape))
        raw = np.empty(n * 3, np.uint8)
        what = EXPORT_SPARSE_K if which == "k" else EXPORT_SPARSE_V
        _check(self._lib.swan_debug_export(self._h, int(layer), what,
                                           raw.ctypes.data_as(ctypes.c_void_p), raw.nbytes),
               "swan_debug_export")
        idx = raw[:n].reshape(shape)
        vals = raw[n:].view(np.float16).reshape(shape)
        return idx, vals

    def export_buffer_seq(self, layer: int, b: int, which: str) -> np.ndarray:
        sp, bf = self.lengths(layer)
        out = np.empty((self.n_kv_heads, bf[b], self.head_dim), np.float16)
        what = EXPORT_BUFFER_K if which == "k" else EXPORT_BUFFER_V
        _check(self._lib.swan_debug_export_seq(self._h, int(layer), int(b), what,
                                               out.ctypes.data_as(ctypes.c_void_p), out.nbytes),
               "swan_debug_export_seq")
        return out

    def export_sparse_seq(self, layer: int, b: int, which: str):
        sp, bf = self.lengths(layer)
        shape = (self.n_kv_heads, sp[b], self.k_store if which == "k" else self.k_store_v)
        n = int(np.prod(shape))
        raw = np.empty(max(1, n * 3), np.uint8)
        what = EXPORT_SPARSE_K if which == "k" else EXPORT_SPARSE_V
        _check(self._lib.swan_debug_export_seq(self._h, int(layer), int(b), what,
                                               raw.ctypes.data_as(ctypes.c_void_p), n * 3),
               "swan_debug_export_seq")
        return raw[:n].reshape(shape), raw[n:n * 3].view(np.float16).reshape(shape)

    def timing_enable(self, on: bool = True):
        _check(self._lib.swan_timing_enable(self._h, 1 if on else 0), "swan_timing_enable")

    def timing_read(self) -> dict:
        t = Timing()
        _check(self._lib.swan_timing_read(self._h, ctypes.byref(t)), "swan_timing_read")
        return {KERNEL_NAMES[k]: (t.ms[k], t.launches[k]) for k in KERNEL_NAMES}

    def launch_count(self) -> int:
        return int(self._lib.swan_launch_count(self._h))


def debug_fail_after(kind: int, n: int):
    """Test hook: the (n+1)-th next device allocation (FAULT_ALLOC) or kernel
    launch (FAULT_LAUNCH) fails on the host; n = -1 turns it off."""
    _check(load_library().swan_debug_fail_after(int(kind), int(n)), "swan_debug_fail_after")


def debug_starve_tc(limit_ns: int):
    """Test hook: the next tensor-core launch issues no copies and its
    barrier waits give up after ``limit_ns`` (``swan_debug_starve_tc``)."""
    _check(load_library().swan_debug_starve_tc(int(limit_ns)), "swan_debug_starve_tc")


def decode_noalloc(view: CacheView, q, out, stream=None):
    """One decode step over a caller-owned cache with no device allocation
    (``swan_decode_noalloc``); ``stream``: a ``torch.cuda.Stream`` or None for
    the current stream."""
    import torch
    lib = load_library()
    if stream is None:
        stream = torch.cuda.current_stream()
    _check(lib.swan_decode_noalloc(ctypes.byref(view), _ptr(q), _ptr(out),
                                   ctypes.c_void_p(stream.cuda_stream)), "swan_decode_noalloc")
    return out


def noalloc_check(stream=None):
    """Raise SwanError if the last ``decode_noalloc`` on this device set its
    device status word (``swan_noalloc_check``; synchronises ``stream``)."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    _check(load_library().swan_noalloc_check(ctypes.c_void_p(stream.cuda_stream)), "swan_noalloc_check")


# ---------------------------------------------------------------------------
# Offline basis construction (swan_basis.h)
# ---------------------------------------------------------------------------

def _stream_handle(stream):
    import torch
    return (stream or torch.cuda.current_stream()).cuda_stream


def rows_of(t, group: int = 1) -> SwanVectors:
    """Vectors that are the contiguous last dimension (128) of a CUDA fp16
    tensor ``[n_mats * group][count][128]`` (e.g. Q ``[N_q][n][d]`` grouped by
    kv head, or K / V ``[N_kv][n][d]``)."""
    if t.dim() != 3 or t.shape[-1] != 128:
        raise ValueError("expected [heads][count][128]")
    if t.shape[0] % group:
        raise ValueError("heads not divisible by group")
    s = t.stride()
    if s[2] != 1:
        raise ValueError("the last dimension must be contiguous")
    v = SwanVectors(_ptr_any(t), t.shape[0] // group, group, t.shape[1], s[0] * group, s[0], s[1], 1)
    v._tensor = t  # the description holds the tensor's memory alive
    return v


def columns_of(w, group: int = 1) -> SwanVectors:
    """Vectors that are the columns of the ``[128][d_model]`` row blocks of a
    CUDA fp16 matrix ``[n_mats * group * 128][d_model]`` (W_O; block h is
    query head h's slice)."""
    if w.dim() != 2 or w.shape[0] % (128 * group):
        raise ValueError("expected [n_mats * group * 128][d_model]")
    if w.stride(1) != 1:
        raise ValueError("rows must be contiguous")
    ld = w.stride(0)
    v = SwanVectors(_ptr_any(w), w.shape[0] // (128 * group), group, w.shape[1], group * 128 * ld, 128 * ld,
                    1, ld)
    v._tensor = w  # the description holds the tensor's memory alive
    return v


def _ptr_any(t) -> int:
    if not t.is_cuda:
        raise ValueError("tensor must live on the GPU")
    return t.data_ptr()


class Gram:
    """Accumulates S^T S of joint matrices on the GPU (swan_gram) into a CUDA
    fp32 tensor ``[n_mats][128][128]``; owns the workspace."""

    def __init__(self, n_mats: int, device=None, stream=None):
        import torch
        self._lib = load_library()
        self.stream = stream
        self.n_mats = n_mats
        self.gram = torch.zeros((n_mats, 128, 128), dtype=torch.float32, device=device or "cuda")
        nbytes = self._lib.swan_gram_workspace_bytes(n_mats)
        self._ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=self.gram.device)
        base = self._ws.data_ptr()
        self._ws_ptr = (base + 255) // 256 * 256
        self._ws_bytes = nbytes

    def add(self, vectors: SwanVectors, accumulate: bool = True):
        if vectors.n_mats != self.n_mats:
            raise ValueError("n_mats differs from the Gram matrices'")
        _check(self._lib.swan_gram(ctypes.byref(vectors), ctypes.c_void_p(self.gram.data_ptr()),
                                   int(accumulate), ctypes.c_void_p(self._ws_ptr), self._ws_bytes,
                                   ctypes.c_void_p(_stream_handle(self.stream))), "swan_gram")
        return self

    def check(self):
        _check(self._lib.swan_basis_check(ctypes.c_void_p(self._ws_ptr),
                                          ctypes.c_void_p(_stream_handle(self.stream))), "swan_basis_check")


def basis_eig(gram, stream=None):
    """Eigenvectors (R, columns by decreasing eigenvalue), eigenvalues and
    sweep counts of CUDA fp32 Gram matrices ``[n][128][128]``."""
    import torch
    lib = load_library()
    n = gram.shape[0]
    R = torch.empty_like(gram)
    lam = torch.empty((n, 128), dtype=torch.float32, device=gram.device)
    sweeps = torch.empty((n,), dtype=torch.int32, device=gram.device)
    _check(lib.swan_basis_eig(ctypes.c_void_p(_ptr(gram)), n, ctypes.c_void_p(R.data_ptr()),
                              ctypes.c_void_p(lam.data_ptr()), ctypes.c_void_p(sweeps.data_ptr()),
                              ctypes.c_void_p(_stream_handle(stream))), "swan_basis_eig")
    return R, lam, sweeps


def energy(vectors: SwanVectors, R, out=None, accumulate: bool = False, stream=None):
    """Energy kept by top-k pruning in the basis R, for k = 0..128: CUDA fp64
    ``[n_mats][129]``."""
    import torch
    lib = load_library()
    if out is None:
        out = torch.zeros((vectors.n_mats, 129), dtype=torch.float64, device=R.device)
    _check(lib.swan_energy(ctypes.byref(vectors), ctypes.c_void_p(_ptr(R)), ctypes.c_void_p(out.data_ptr()),
                           int(accumulate), ctypes.c_void_p(_stream_handle(stream))), "swan_energy")
    return out
