"""Python binding of libmone.so (MoNe test-time learning on one GB300 GPU).

Argument marshalling only: every function below forwards to the C entry point
of the same name declared in ``include/mone.h``; all arithmetic runs in the
library's CUDA kernels.  PyTorch tensors are accepted for device buffers (their
``data_ptr()`` is passed) and the current torch CUDA stream is used when no
stream is given.  There is no fallback: if ``libmone.so`` is missing or cannot
be loaded, ``lib()`` raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

_PKG = os.path.dirname(os.path.abspath(__file__))
# MONE_LIB selects another build of the library, e.g. the MONE_DEBUG build (libmone_debug.so)
LIB_PATH = os.environ.get("MONE_LIB") or os.path.join(_PKG, "libmone.so")
DEBUG_LIB_PATH = os.path.join(_PKG, "libmone_debug.so")

MONE_FP32, MONE_BF16 = 0, 1
MONE_PLAIN, MONE_PAPER = 0, 1
MONE_LOSS_DOT, MONE_LOSS_MSE = 0, 1
MONE_MEM_MLP, MONE_MEM_SWIGLU = 0, 1
MONE_RENORM_ROWS, MONE_RENORM_OUT = 0, 1
MONE_GATE_LINEAR, MONE_GATE_SILU = 0, 1

STATUS = {0: "MONE_OK", 1: "MONE_ERR_INVALID_ARG", 2: "MONE_ERR_UNSUPPORTED_SHAPE", 3: "MONE_ERR_OOM",
          4: "MONE_ERR_CUDA", 5: "MONE_ERR_TIMEOUT", 6: "MONE_ERR_NONFINITE", 7: "MONE_ERR_UNSUPPORTED",
          8: "MONE_ERR_CHECK"}

# Every symbol include/mone.h declares.
EXPORTS = ("mone_mem_init", "mone_ttl_segment", "mone_ttl_context", "mone_mem_generate_kv", "mone_mem_free",
           "mone_mem_read_state", "mone_mem_write_state", "mone_mem_sync", "mone_mem_launch_count",
           "mone_status_string", "mone_abi_version", "mone_mem_set_timing", "mone_mem_kernel_time",
           "mone_last_error", "mone_mem_generate_kv_noalloc", "mone_attention", "mone_mem_kernel_busy",
           "mone_ttl_context_metrics", "mone_ttl_context_host")

KERNEL_KINDS = ("prepass", "phase_a", "phase_b", "finalize", "read", "mse", "attention", "resident", "stage")


class MoneError(RuntimeError):
    def __init__(self, fn: str, code: int, detail: str = ""):
        self.code = code
        super().__init__(f"{fn} failed: {STATUS.get(code, code)}" + (f" ({detail})" if detail else ""))


class mone_config(ctypes.Structure):
    _fields_ = [("n_ctx", ctypes.c_int), ("n_layers", ctypes.c_int), ("d_in", ctypes.c_int),
                ("d_hid", ctypes.c_int), ("d_out", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("seg_T", ctypes.c_int), ("dtype", ctypes.c_int),
                ("mode", ctypes.c_int), ("lr", ctypes.c_float), ("rms_eps", ctypes.c_float), ("loss", ctypes.c_int),
                ("memory", ctypes.c_int), ("mem_heads", ctypes.c_int), ("renorm_axis", ctypes.c_int),
                ("gate_act", ctypes.c_int)]


class mone_meta(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("alpha", "gamma", "w_eta", "b_eta", "w_beta", "b_beta", "gate")]


_lib = None


def lib(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libmone.so (once).  Raises OSError when it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise OSError(f"libmone.so not found at {p}; build it with paper_2608_17616_gb300.build.build()")
    L = ctypes.CDLL(p)
    vp, i, ll, f = ctypes.c_void_p, ctypes.c_int, ctypes.c_longlong, ctypes.c_float
    sig = {
        "mone_mem_init": ([ctypes.POINTER(mone_config), vp, vp, ctypes.POINTER(mone_meta), vp,
                           ctypes.POINTER(vp)], i),
        "mone_ttl_segment": ([vp, i, i, vp, vp, vp, i, vp, vp, vp], i),
        "mone_ttl_context": ([vp, vp, vp, vp, ll, vp], i),
        "mone_ttl_context_metrics": ([vp, vp, vp, vp, ll, vp, vp, vp], i),
        "mone_ttl_context_host": ([vp, vp, vp, vp, ll, ll, vp], i),
        "mone_mem_generate_kv": ([vp, vp, i, vp, vp, ctypes.POINTER(ll), vp], i),
        "mone_mem_generate_kv_noalloc": ([vp, vp, i, vp, vp, ctypes.POINTER(ll), vp], i),
        "mone_attention": ([vp, vp, i, i, vp, vp, ctypes.POINTER(ll), i, vp, vp], i),
        "mone_mem_free": ([vp], i),
        "mone_mem_read_state": ([vp, vp, vp, vp, vp, vp], i),
        "mone_mem_write_state": ([vp, vp, vp, vp, vp, vp], i),
        "mone_mem_sync": ([vp, vp], i),
        "mone_mem_launch_count": ([vp], ll),
        "mone_status_string": ([i], ctypes.c_char_p),
        "mone_abi_version": ([], i),
        "mone_last_error": ([], ctypes.c_char_p),
        "mone_mem_set_timing": ([vp, i], i),
        "mone_mem_kernel_time": ([vp, i, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ll)], i),
        "mone_mem_kernel_busy": ([vp, i, ctypes.POINTER(ctypes.c_double)], i),
    }
    for name, (args, res) in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = res
    if path is None:
        _lib = L
    return L


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn: str, rc: int):
    if rc != 0:
        detail = lib().mone_last_error().decode() if rc in (3, 4, 8) else ""
        raise MoneError(fn, rc, detail)


def make_config(n_ctx, n_layers, d_in, d_hid, d_out, n_kv_heads, head_dim, seg_T, dtype, mode, lr,
                rms_eps=1e-6, loss=0, memory=0, mem_heads=1, renorm_axis=0, gate_act=0) -> mone_config:
    return mone_config(n_ctx, n_layers, d_in, d_hid, d_out, n_kv_heads, head_dim, seg_T, dtype, mode, lr, rms_eps,
                       loss, memory, mem_heads, renorm_axis, gate_act)


def make_meta(meta: Optional[dict]) -> Optional[mone_meta]:
    """mone_meta from a dict of device fp32 tensors (keys as in the header)."""
    if meta is None:
        return None
    return mone_meta(*[_ptr(meta.get(k)) for k in ("alpha", "gamma", "w_eta", "b_eta", "w_beta", "b_beta", "gate")])


def mone_mem_init(cfg: mone_config, W1_0, W2_0, meta=None, stream=None) -> int:
    h = ctypes.c_void_p()
    m = make_meta(meta) if isinstance(meta, dict) else meta
    rc = lib().mone_mem_init(ctypes.byref(cfg), _ptr(W1_0), _ptr(W2_0), ctypes.byref(m) if m is not None else None,
                             _stream(stream), ctypes.byref(h))
    _check("mone_mem_init", rc)
    return h.value


def mone_ttl_segment(h: int, ctx: int, layer: int, X, K, V, n_tok: int, eta=None, loss_out=None, stream=None):
    _check("mone_ttl_segment", lib().mone_ttl_segment(h, ctx, layer, _ptr(X), _ptr(K), _ptr(V), n_tok, _ptr(eta),
                                                      _ptr(loss_out), _stream(stream)))


def mone_ttl_context(h: int, X, K, V, N: int, stream=None):
    _check("mone_ttl_context", lib().mone_ttl_context(h, _ptr(X), _ptr(K), _ptr(V), N, _stream(stream)))


def mone_ttl_context_metrics(h: int, X, K, V, N: int, seg_loss=None, seg_step=None, stream=None):
    """mone_ttl_context with per-segment loss and squared step norm ([S][C] fp32 device buffers)."""
    _check("mone_ttl_context_metrics", lib().mone_ttl_context_metrics(h, _ptr(X), _ptr(K), _ptr(V), N, _ptr(seg_loss),
                                                                      _ptr(seg_step), _stream(stream)))


def mone_ttl_context_host(h: int, X, K, V, N: int, chunk_tokens: int = 0, stream=None):
    """mone_ttl_context over host tensors (pinned CPU tensors, or host memory the device reads through
    the host's page tables): the library stages chunks of whole segments into its device windows."""
    _check("mone_ttl_context_host", lib().mone_ttl_context_host(h, _ptr(X), _ptr(K), _ptr(V), N, chunk_tokens,
                                                                _stream(stream)))


def mone_mem_generate_kv(h: int, Xq, Q: int, K_out, V_out, strides: Sequence[int], stream=None):
    arr = (ctypes.c_longlong * 4)(*[int(s) for s in strides])
    _check("mone_mem_generate_kv", lib().mone_mem_generate_kv(h, _ptr(Xq), Q, _ptr(K_out), _ptr(V_out), arr,
                                                              _stream(stream)))


def mone_mem_generate_kv_noalloc(h: int, Xq, Q: int, K_out, V_out, strides: Sequence[int], stream=None):
    """The memory read without any device allocation (fixed 16 MiB library scratch)."""
    arr = (ctypes.c_longlong * 4)(*[int(s) for s in strides])
    _check("mone_mem_generate_kv_noalloc", lib().mone_mem_generate_kv_noalloc(h, _ptr(Xq), Q, _ptr(K_out),
                                                                              _ptr(V_out), arr, _stream(stream)))


def mone_attention(h: int, Q, n_q_heads: int, Lq: int, K, V, kv_strides: Sequence[int], n_mem: int, out,
                   stream=None):
    """Consumer attention of the read (Eq. 5): query tokens over [memory tokens || their own keys]."""
    arr = (ctypes.c_longlong * 4)(*[int(s) for s in kv_strides])
    _check("mone_attention", lib().mone_attention(h, _ptr(Q), n_q_heads, Lq, _ptr(K), _ptr(V), arr, n_mem, _ptr(out),
                                                  _stream(stream)))


def mone_mem_free(h: int):
    _check("mone_mem_free", lib().mone_mem_free(h))


def mone_mem_read_state(h: int, W1=None, W2=None, mu1=None, mu2=None, stream=None):
    _check("mone_mem_read_state", lib().mone_mem_read_state(h, _ptr(W1), _ptr(W2), _ptr(mu1), _ptr(mu2),
                                                            _stream(stream)))


def mone_mem_write_state(h: int, W1=None, W2=None, mu1=None, mu2=None, stream=None):
    _check("mone_mem_write_state", lib().mone_mem_write_state(h, _ptr(W1), _ptr(W2), _ptr(mu1), _ptr(mu2),
                                                              _stream(stream)))


def mone_mem_sync(h: int, stream=None):
    _check("mone_mem_sync", lib().mone_mem_sync(h, _stream(stream)))


def mone_mem_launch_count(h: int) -> int:
    return lib().mone_mem_launch_count(h)


def mone_status_string(code: int) -> str:
    return lib().mone_status_string(code).decode()


def mone_abi_version() -> int:
    return lib().mone_abi_version()


def mone_last_error() -> str:
    return lib().mone_last_error().decode()


def mone_mem_set_timing(h: int, enable: bool):
    _check("mone_mem_set_timing", lib().mone_mem_set_timing(h, 1 if enable else 0))


def mone_mem_kernel_time(h: int, kind: int):
    """(total device ms, launches) of one kernel kind since timing was enabled."""
    ms = ctypes.c_double()
    n = ctypes.c_longlong()
    _check("mone_mem_kernel_time", lib().mone_mem_kernel_time(h, kind, ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def mone_mem_kernel_busy(h: int, kind: int) -> float:
    """Busy time (ms) of one kernel kind since timing was enabled: the union of its launches'
    event intervals, overlapping launches counted once."""
    ms = ctypes.c_double()
    _check("mone_mem_kernel_busy", lib().mone_mem_kernel_busy(h, kind, ctypes.byref(ms)))
    return ms.value


def kv_strides(n_layers: int, n_kv: int, Q: int, head_dim: int):
    """Element strides (ctx, layer, kv_head, q) of a dense [n_ctx][n_layers][n_kv][Q][head_dim] output."""
    return (n_layers * n_kv * Q * head_dim, n_kv * Q * head_dim, Q * head_dim, head_dim)
