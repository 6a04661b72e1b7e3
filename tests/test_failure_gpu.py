"""Failure paths, exercised without faulting or hanging a GPU.

reskv_test_inject makes (a) the next decode launch's warps (or, in a build,
the persistent Lloyd assignment's CTA 0 certifier) give up their first wait
as a timed-out bounded wait would -- the kernel sets its status word, waits
for its own copies in flight and returns -- and (b) the n-th device
allocation fail as cudaMalloc out of memory would.  The host must see the
fault (reskv_check_status: RESKV_ERR_DEVICE_STATUS; the call: RESKV_ERR_OOM),
leave the output handle untouched, leak no device memory, and a fresh handle
must decode correctly afterwards.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import assert_output_parity
from test_decode_gpu import SPLITS, oracle_decode_all, queries_for, synthetic_layout

pytestmark = pytest.mark.gpu

KERNELS = {"fma": R.RESKV_DECODE_FMA, "mma": R.RESKV_DECODE_MMA,
           "cluster": R.RESKV_DECODE_CLUSTER, "lse": R.RESKV_DECODE_LSE_MERGE}


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


@pytest.fixture(autouse=True)
def no_pending_injection():
    yield
    R.reskv_test_inject(R.RESKV_TEST_FAIL_FIRST_WAIT, 0)
    R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, 0)


def _case(kernel):
    L, Bt, H, G, b = 2, 3, 2, 4, 300
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b, decode_kernel=KERNELS[kernel])
    return w, lay, cfg, queries_for(w, L, Bt, H, G)


@pytest.mark.parametrize("kernel", list(KERNELS))
@pytest.mark.parametrize("layer", [-1, 1])
def test_timed_out_wait_is_reported_and_a_fresh_handle_decodes(kernel, layer):
    w, lay, cfg, Q = _case(kernel)
    h = R.reskv_import_cache(cfg, **lay)
    Qd = (Q if layer < 0 else Q[layer]).cuda().contiguous()
    O = torch.zeros(Qd.shape, dtype=torch.float32, device="cuda")
    R.reskv_test_inject(R.RESKV_TEST_FAIL_FIRST_WAIT, 1)
    R.reskv_decode_attn(h, layer, Qd, O)              # the launch itself succeeds
    torch.cuda.synchronize()
    with pytest.raises(R.ReskvError) as e:
        R.reskv_check_status(h)
    assert e.value.status == R.RESKV_ERR_DEVICE_STATUS and "word 1" in str(e.value)
    h.free()
    # the context stays usable: a fresh handle decodes correctly
    h2 = R.reskv_import_cache(cfg, **lay)
    O2 = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(h2, layer, Qd, O2)
    torch.cuda.synchronize()
    R.reskv_check_status(h2)
    ref = oracle_decode_all(lay, Q, cfg)
    assert_output_parity(O2.cpu().numpy(), ref if layer < 0 else ref[layer], kernel)
    h2.free()


def test_timed_out_wait_in_construction_is_reported_and_a_fresh_build_matches():
    """The persistent Lloyd assignment (Alg. 1): CTA 0's certifier gives up its
    first wait as a timed-out bounded wait would.  Every role of that CTA
    leaves at a tile boundary, its copies and MMAs finish, the build returns
    with the timeout in the status word, the later construction kernels stay
    inside their arrays, and a fresh build matches the oracle."""
    import re

    from test_build_gpu import lib_config, make_inputs, run_case

    w = wl.WORKLOADS["tiny"]                      # one unit, r = 32: the persistent form
    _, (Kd, Vd, Qdv) = make_inputs(w)
    cfg = lib_config(w)
    R.reskv_test_inject(R.RESKV_TEST_FAIL_FIRST_WAIT, 1)
    cache = R.reskv_build_cache(cfg, Kd, Vd, Qdv if w.n_obs > 0 else None)
    torch.cuda.synchronize()
    with pytest.raises(R.ReskvError) as e:
        R.reskv_check_status(cache)
    assert e.value.status == R.RESKV_ERR_DEVICE_STATUS
    m = re.search(r"word (\d+)", str(e.value))
    assert m and int(m.group(1)) & 1                 # kStatusWaitTimeout
    cache.free()
    out = run_case(w)                                  # a fresh build: full parity
    assert out["worst_rel"] < 2e-3


def _raw_build(cfg, Ks, Vs, Qs):
    """reskv_build_cache through ctypes with a sentinel in *out."""
    L = cfg.n_layers
    kp = (ctypes.c_void_p * L)(*[k.data_ptr() for k in Ks])
    vp = (ctypes.c_void_p * L)(*[v.data_ptr() for v in Vs])
    qp = (ctypes.c_void_p * L)(*[q.data_ptr() for q in Qs])
    out = ctypes.c_void_p(0x5e771e)
    st = R.load_library().reskv_build_cache(ctypes.byref(cfg), kp, vp, qp,
                                            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream),
                                            ctypes.byref(out))
    return st, out


def _free_bytes():
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def test_allocation_failures_in_build_leave_nothing_behind():
    """Every device allocation of reskv_build_cache in turn fails: the call
    returns RESKV_ERR_OOM, *out keeps its value, and the device holds as much
    free memory as before the call."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=1024, budget=256, batch=1,
                  n_kv_heads=2, n_layers=2)
    Ks, Vs, Qs = [], [], []
    for l in range(w.n_layers):
        K, V, Qo, _ = wl.layer_inputs(w, l, "cuda")
        Ks.append(K)
        Vs.append(V)
        Qs.append(Qo)
    cfg = R.reskv_config_default(batch=w.batch, n_layers=w.n_layers, n_kv_heads=w.n_kv_heads,
                                 group=w.group, seq_len=w.seq_len, budget=w.budget,
                                 n_obs=w.n_obs, n_fit=w.n_fit, n_val=w.n_val, keep_debug=1)
    st, out = _raw_build(cfg, Ks, Vs, Qs)               # warm: module loads, attributes
    assert st == R.RESKV_OK
    R.load_library().reskv_free(out)
    free0 = _free_bytes()
    failed = 0
    for n in range(1, 200):
        R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, n)
        st, out = _raw_build(cfg, Ks, Vs, Qs)
        if st == R.RESKV_OK:                            # past the last allocation
            R.load_library().reskv_free(out)
            break
        assert st == R.RESKV_ERR_OOM, (n, st, R.reskv_last_error())
        assert out.value == 0x5e771e, n
        assert _free_bytes() == free0, f"allocation {n}: device memory leaked"
        failed += 1
    R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, 0)
    assert failed >= 10, failed                         # the layout and the scratch arrays
    assert _free_bytes() == free0


def test_allocation_failures_in_import_and_host_staging():
    w, lay, cfg, Q = _case("mma")
    h = R.reskv_import_cache(cfg, **lay)                # warm
    h.free()
    free0 = _free_bytes()
    failed = 0
    for n in range(1, 100):
        R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, n)
        try:
            h = R.reskv_import_cache(cfg, **lay)
        except R.ReskvError as e:
            assert e.status == R.RESKV_ERR_OOM, (n, str(e))
            assert _free_bytes() == free0, f"allocation {n}: device memory leaked"
            failed += 1
            continue
        h.free()
        break
    R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, 0)
    assert failed >= 8
    # pageable host buffers are staged through buffers made on first use
    h = R.reskv_import_cache(cfg, **lay)
    Qh = Q.contiguous()
    Oh = torch.empty(Q.shape, dtype=torch.float32)
    R.reskv_test_inject(R.RESKV_TEST_FAIL_ALLOC, 2)     # the output staging buffer
    with pytest.raises(R.ReskvError) as e:
        R.reskv_decode_attn_host(h, Qh, Oh)
    assert e.value.status == R.RESKV_ERR_OOM
    R.reskv_decode_attn_host(h, Qh, Oh)                 # staging made now; works
    torch.cuda.synchronize()
    assert_output_parity(Oh.numpy(), oracle_decode_all(lay, Q, cfg), "staged after OOM")
    h.free()
