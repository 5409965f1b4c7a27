"""C-ABI checks that need no GPU: the library loads, exports every symbol the
header declares, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

import paper_2608_17616_gb300 as mone
from paper_2608_17616_gb300 import build as mbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    mbuild.build()
    return mone.lib()


def header_functions():
    text = open(os.path.join(ROOT, "include", "mone.h")).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?(?:\w+\**\s+)+\**(mone_\w+)\(", text, re.M)))


def test_header_declares_the_boundary():
    names = header_functions()
    for required in ("mone_mem_init", "mone_ttl_segment", "mone_ttl_context", "mone_mem_generate_kv",
                     "mone_mem_free"):
        assert required in names
    assert set(names) == set(mone.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    raw = ctypes.CDLL(mone.LIB_PATH)
    for name in header_functions():
        assert hasattr(raw, name), name
    assert L.mone_abi_version() == 7


def test_status_strings(L):
    for code in range(9):
        assert mone.mone_status_string(code)
    assert mone.mone_status_string(0) == "ok"


def cfg(**kw):
    base = dict(n_ctx=1, n_layers=2, d_in=256, d_hid=256, d_out=256, n_kv_heads=2, head_dim=64, seg_T=128,
                dtype=mone.MONE_BF16, mode=mone.MONE_PLAIN, lr=1e-2)
    base.update(kw)
    return mone.make_config(**base)


def init_rc(L, c, w1=16, w2=16, meta=None):
    h = ctypes.c_void_p()
    return L.mone_mem_init(ctypes.byref(c) if c is not None else None, w1, w2, meta, None, ctypes.byref(h))


def test_init_rejects_bad_arguments_without_a_device(L):
    assert init_rc(L, None) == 1
    assert init_rc(L, cfg(), w1=None) == 1
    assert init_rc(L, cfg(), w1=8) == 1                     # misaligned
    assert init_rc(L, cfg(dtype=7)) == 1
    assert init_rc(L, cfg(mode=3)) == 1
    assert init_rc(L, cfg(n_layers=0)) == 1
    assert init_rc(L, cfg(lr=float("nan"))) == 1
    assert init_rc(L, cfg(mode=mone.MONE_PAPER)) == 1         # paper mode needs meta-parameters
    assert init_rc(L, cfg(loss=2)) == 1                         # no such loss


def test_swiglu_memory_validation(L):
    sw = dict(d_in=896, d_hid=224, d_out=896, n_kv_heads=7, head_dim=64, seg_T=128, memory=mone.MONE_MEM_SWIGLU,
              mem_heads=4)
    assert init_rc(L, cfg(memory=2)) == 1                                  # no such memory form
    assert init_rc(L, cfg(**{**sw, "mem_heads": 3})) == 1                 # d_in not split evenly into heads
    assert init_rc(L, cfg(**{**sw, "dtype": mone.MONE_FP32})) == 7        # tensor-core path only
    assert init_rc(L, cfg(**{**sw, "loss": mone.MONE_LOSS_MSE})) == 7     # Eq. 7 loss only
    assert init_rc(L, cfg(**{**sw, "d_hid": 300})) == 2                   # hidden units per head <= 256
    assert init_rc(L, cfg(**{**sw, "mem_heads": 2})) == 2                 # dh = 448 > 256
    assert init_rc(L, cfg(**{**sw, "d_out": 768, "n_kv_heads": 6})) == 2  # output width must equal d_in
    assert init_rc(L, cfg(**{**sw, "lr": float("inf")})) == 1             # rates checked for every memory form
    assert init_rc(L, cfg(**{**sw, "rms_eps": float("nan")})) == 1


def test_renorm_axis_and_gate_validation(L):
    assert init_rc(L, cfg(renorm_axis=2)) == 1                  # no such renormalisation axis
    assert init_rc(L, cfg(gate_act=2)) == 1                     # no such gate activation
    sw = dict(d_in=896, d_hid=224, d_out=896, n_kv_heads=7, head_dim=64, seg_T=128, memory=mone.MONE_MEM_SWIGLU,
              mem_heads=4)
    assert init_rc(L, cfg(**{**sw, "renorm_axis": mone.MONE_RENORM_OUT})) == 7  # output channels: MLP only


def test_squared_error_loss_passes_validation_on_both_paths(L):
    # the squared-error variant runs on both paths (MLP memory).  The configuration is checked
    # before the weight pointers, so a misaligned W1_0 (argument error, no device work) shows
    # that the configuration itself was accepted
    for dtype in (mone.MONE_FP32, mone.MONE_BF16):
        assert init_rc(L, cfg(dtype=dtype, loss=mone.MONE_LOSS_MSE), w1=8) == 1
    # (an unsupported configuration still answers 7 with the same misaligned pointer)
    assert init_rc(L, cfg(memory=mone.MONE_MEM_SWIGLU, d_in=896, d_hid=224, d_out=896, n_kv_heads=7, mem_heads=4,
                          loss=mone.MONE_LOSS_MSE), w1=8) == 7


def test_init_rejects_unsupported_shapes(L):
    assert init_rc(L, cfg(head_dim=96, d_out=384, n_kv_heads=2)) == 2
    assert init_rc(L, cfg(d_out=512)) == 2                    # d_out != 2 * n_kv * hd
    assert init_rc(L, cfg(d_in=192)) == 2                     # bf16 tiles are 128 wide
    assert init_rc(L, cfg(d_hid=384)) == 2                    # bf16 hidden tiles are 256 wide
    assert init_rc(L, cfg(seg_T=192)) == 2
    assert init_rc(L, cfg(seg_T=8192)) == 2
    assert init_rc(L, cfg(dtype=mone.MONE_FP32, d_in=96)) == 2


def test_calls_on_invalid_handles(L):
    bogus = 0x1000
    assert L.mone_mem_free(None) == 1
    assert L.mone_mem_free(bogus) == 1
    assert L.mone_ttl_context(bogus, 16, 16, 16, 128, None) == 1
    assert L.mone_ttl_segment(bogus, 0, 0, 16, 16, 16, 1, None, None, None) == 1
    arr = (ctypes.c_longlong * 4)(0, 0, 0, 0)
    assert L.mone_mem_generate_kv(bogus, 16, 1, 16, 16, arr, None) == 1
    assert L.mone_mem_sync(bogus, None) == 1
    assert L.mone_mem_launch_count(bogus) == -1
    assert L.mone_ttl_context_host(bogus, 16, 16, 16, 128, 0, None) == 1
    assert L.mone_ttl_context_metrics(bogus, 16, 16, 16, 128, None, None, None) == 1
    assert L.mone_attention(bogus, 16, 2, 4, 16, 16, arr, 0, 16, None) == 1


@pytest.mark.skipif(os.path.exists("/dev/nvidia0"), reason="checks the behaviour on a machine without a GPU")
def test_init_without_gpu_fails_loudly(L):
    # valid arguments, no device: the library reports a CUDA error, it never falls back to the CPU
    assert init_rc(L, cfg()) == 4


def test_debug_build_compiles_and_exports_every_symbol():
    # the MONE_DEBUG variant (device-side index checks) cross-compiles for sm_103a and exports
    # the same boundary; its checks run on a GPU in tests/test_debug_build_gpu.py
    from paper_2608_17616_gb300 import build
    path = build.build(debug=True)
    assert path.endswith("libmone_debug.so")
    raw = ctypes.CDLL(path)
    for name in header_functions():
        assert hasattr(raw, name), name
    raw.mone_abi_version.restype = ctypes.c_int
    assert raw.mone_abi_version() == 7
