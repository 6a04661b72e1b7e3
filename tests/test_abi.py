"""The C ABI library loads and exports what include/reskv.h declares (no GPU).

Only host-side paths run here: symbol lookup, struct layout, defaults and
argument validation that fails before any CUDA call.
"""
import ctypes
import os
import re
import subprocess
import tempfile

import pytest

from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "reskv.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return R.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(reskv_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert "reskv_build_cache" in names and "reskv_decode_attn" in names and "reskv_free" in names
    for n in names:
        assert hasattr(lib, n), f"{n} declared in reskv.h but not exported"
    out = subprocess.run(["nm", "-D", "--defined-only", R.LIB_PATH], capture_output=True,
                         text=True).stdout
    exported = set(re.findall(r"\bT (reskv_[a-z_]+)", out))
    assert set(names) <= exported


def test_struct_layout_matches_c(lib, tmp_path):
    """ctypes mirrors of the ABI structs have the C compiler's size and offsets."""
    src = tmp_path / "layout.c"
    fields = [f for f, _ in R.reskv_config._fields_]
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "reskv.h"', "int main(void){",
             'printf("%zu\\n", sizeof(reskv_config));',
             'printf("%zu\\n", sizeof(reskv_host_cache));',
             'printf("%zu\\n", sizeof(reskv_cache_info));']
    lines += [f'printf("%zu\\n", offsetof(reskv_config, {f}));' for f in fields]
    lines += ['printf("%zu\\n", sizeof(reskv_device_cache));']
    lines += [f'printf("%zu\\n", offsetof(reskv_device_cache, {f}));'
              for f, _ in R.reskv_device_cache._fields_]
    lines += ["return 0;}"]
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)],
                   check=True)
    vals = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True,
                                           check=True).stdout.split()]
    assert vals[0] == ctypes.sizeof(R.reskv_config)
    assert vals[1] == ctypes.sizeof(R.reskv_host_cache)
    assert vals[2] == ctypes.sizeof(R.reskv_cache_info)
    for f, off in zip(fields, vals[3:3 + len(fields)]):
        assert getattr(R.reskv_config, f).offset == off, f
    dfields = [f for f, _ in R.reskv_device_cache._fields_]
    assert vals[3 + len(fields)] == ctypes.sizeof(R.reskv_device_cache)
    for f, off in zip(dfields, vals[4 + len(fields):]):
        assert getattr(R.reskv_device_cache, f).offset == off, f


def test_defaults_are_the_papers(lib):
    cfg = R.reskv_config_default()
    assert (cfg.recent_window, cfg.n_fit, cfg.n_val, cfg.pool_kernel, cfg.lloyd_iters) == (64, 96, 32, 5, 4)
    assert [round(cfg.grid_ratios[i], 6) for i in range(cfg.n_grid)] == [0.0, 0.05, 0.1, 0.15, 0.2]
    assert cfg.delta == pytest.approx(0.01) and cfg.beta == 1.0
    assert cfg.tau == 0.25 and cfg.alpha == 12.0 and cfg.g_min == 0.0
    assert cfg.gate_mode == R.RESKV_GATE_DYNAMIC and cfg.head_dim == 128
    assert cfg.softmax_mode == R.RESKV_SOFTMAX_SHARED and cfg.decode_kernel == R.RESKV_DECODE_AUTO


def test_host_validation_errors(lib):
    st = lib.reskv_decode_attn(None, 0, None, None, None)
    assert st == 1 and "NULL" in R.reskv_last_error()
    cfg = R.reskv_config_default(batch=1, n_layers=1, n_kv_heads=1, seq_len=64, budget=16,
                                 head_dim=64)
    out = ctypes.c_void_p()
    st = lib.reskv_build_cache(ctypes.byref(cfg), (ctypes.c_void_p * 1)(1), (ctypes.c_void_p * 1)(1),
                               None, None, ctypes.byref(out))
    assert st == 2 and "head_dim" in R.reskv_last_error()
    cfg.head_dim = 128
    cfg.group = 3
    st = lib.reskv_build_cache(ctypes.byref(cfg), (ctypes.c_void_p * 1)(1), (ctypes.c_void_p * 1)(1),
                               None, None, ctypes.byref(out))
    assert st == 2 and out.value is None
    cfg.group = 4
    for field, bad, word in (("softmax_mode", 2, "softmax_mode"), ("decode_kernel", 5, "decode_kernel"),
                             ("decode_warps", -1, "decode_warps")):
        setattr(cfg, field, bad)
        st = lib.reskv_build_cache(ctypes.byref(cfg), (ctypes.c_void_p * 1)(1),
                                   (ctypes.c_void_p * 1)(1), None, None, ctypes.byref(out))
        assert st == 1 and word in R.reskv_last_error() and out.value is None, field
        setattr(cfg, field, 0)
    lib.reskv_free(None)                       # NULL-safe


def test_noalloc_binding_checks_every_shape(lib):
    """The no-allocation decode's binding checks every array against the
    shape the kernel will read and write, before any CUDA call: a short
    vslots, logc, n_main, n_res, Q or O raises ValueError naming it."""
    import torch
    U, b, H, G = 16, 32, 4, 4
    good = dict(kslots=torch.zeros((U, b, 128), dtype=torch.bfloat16),
                vslots=torch.zeros((U, b, 128), dtype=torch.bfloat16),
                logc=torch.zeros((U, b), dtype=torch.float32),
                n_main=torch.ones(U, dtype=torch.int32), n_res=torch.zeros(U, dtype=torch.int32),
                Q=torch.zeros((U // H, H * G, 128), dtype=torch.bfloat16),
                O=torch.zeros((U // H, H * G, 128), dtype=torch.float32))

    def call(**over):
        a = dict(good, **over)
        R.reskv_decode_attn_noalloc(a["kslots"], a["vslots"], a["logc"], a["n_main"], a["n_res"],
                                    H, G, a["Q"], a["O"])

    bad = {"vslots": torch.zeros((U, b - 1, 128), dtype=torch.bfloat16),
           "logc": torch.zeros((U - 1, b), dtype=torch.float32),
           "n_main": torch.ones(U - 1, dtype=torch.int32),
           "n_res": torch.zeros(U + 1, dtype=torch.int32),
           "Q": torch.zeros((U // H, H * G - 1, 128), dtype=torch.bfloat16),
           "O": torch.zeros((U // H - 1, H * G, 128), dtype=torch.float32)}
    for name, t in bad.items():
        with pytest.raises(ValueError, match=name):
            call(**{name: t})
    with pytest.raises(ValueError, match="kslots"):
        call(kslots=torch.zeros((U, b, 64), dtype=torch.bfloat16))
    with pytest.raises(ValueError, match="multiple of n_kv_heads"):
        R.reskv_decode_attn_noalloc(*(torch.zeros((U + 1, b, 128), dtype=torch.bfloat16),) * 2,
                                    good["logc"], good["n_main"], good["n_res"], H, G, good["Q"],
                                    good["O"])
    # shapes right: only now the device check (these are host tensors)
    with pytest.raises(ValueError, match="CUDA tensor"):
        call()


def test_fault_injection_arguments_are_checked(lib):
    """reskv_test_inject validates its arguments on the host (no GPU needed)."""
    with pytest.raises(R.ReskvError) as e:
        R.reskv_test_inject(7, 1)
    assert e.value.status == R.RESKV_ERR_INVALID_ARG
    with pytest.raises(R.ReskvError) as e:
        R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, -1)
    assert e.value.status == R.RESKV_ERR_INVALID_ARG
    R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, 0)
    R.reskv_test_inject(R.RESKV_TEST_FAIL_FIRST_WAIT, 0)
