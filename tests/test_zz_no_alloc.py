"""The decode entry point that allocates nothing (reskv_decode_attn_noalloc).

It serves callers that cannot allocate GPU memory while decoding -- for
instance code living inside a host application whose memory manager owns all
device allocations, or latency-critical paths that must avoid cudaMalloc.  They
keep the cache in their own device memory; the library takes its per-call
scratch from a fixed static array instead of allocating.  The output must
agree with the regular entry point (reskv_decode_attn on a handle holding the
same cache), call after call, since every call reuses the same scratch, and
with the fp64 oracle's decode (Alg. 2) of every unit.  After every call the
status readback (reskv_noalloc_check_status) must report no fault and name
the kernel the call took; a fault injected into one call must be reported
once and not disturb the next call.

This file is named so that pytest collects it last; it needs nothing from the
other tests and runs alone in a fresh process as well.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import (assert_output_parity, bf16_bits, bf16_to_f64, empty_layout, errors,
                     unit_from_layout)

pytestmark = pytest.mark.gpu


def _layout(L, Bt, H, b, seed=7):
    """A ragged cache of seeded generator rows (main, residual, unused tail)."""
    U = L * Bt * H
    w = wl.Workload("noalloc", L, Bt, H, 4, 128, b + 32, b, 0, 0, 0, 0, "fixed:0", 1)
    lay = empty_layout(U, b)
    rng = np.random.default_rng(seed)
    for u in range(U):
        l, rem = divmod(u, Bt * H)
        bb, h = divmod(rem, H)
        m = int(rng.integers(1, b + 1))
        r = int(rng.integers(0, b - m + 1))
        K, V = wl.unit_kv(w, l, bb, h)
        lay["n_main"][u], lay["n_res"][u] = m, r
        lay["kslots"][u, :m + r] = bf16_bits(K[:m + r])
        lay["vslots"][u, :m + r] = bf16_bits(V[:m + r])
        if r:
            c = rng.integers(0, 100, r)
            with np.errstate(divide="ignore"):
                lay["logc"][u, m:m + r] = np.log(c.astype(np.float64)).astype(np.float32)
    Q = torch.empty((L, Bt, H * 4, 128), dtype=torch.bfloat16)
    for l in range(L):
        for bb in range(Bt):
            for h in range(H):
                K, _ = wl.unit_kv(w, l, bb, h)
                Q[l, bb, h * 4:(h + 1) * 4] = wl.unit_decode_queries(w, l, bb, h, K, 1)[:, 0]
    return lay, Q


def _oracle(lay, Q):
    """fp64 oracle decode (Alg. 2, dynamic gate) of every unit: [L, B, H*4, 128]."""
    L, Bt, Hq, d = Q.shape
    H = Hq // 4
    qf = bf16_to_f64(Q)
    out = np.zeros(Q.shape)
    cfg = orc.OracleConfig(budget=1)
    for l in range(L):
        for bb in range(Bt):
            for h in range(H):
                u = (l * Bt + bb) * H + h
                out[l, bb, h * 4:(h + 1) * 4] = orc.decode_unit(
                    unit_from_layout(lay, u), qf[l, bb, h * 4:(h + 1) * 4], cfg)
    return out


def _device_arrays(lay, logc=None):
    dev = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).cuda().view(dt)
    return (dev(lay["kslots"].view(np.int16), torch.bfloat16),
            dev(lay["vslots"].view(np.int16), torch.bfloat16),
            dev(lay["logc"], torch.float32) if logc is None else logc,
            dev(lay["n_main"], torch.int32), dev(lay["n_res"], torch.int32))


@pytest.mark.parametrize("b", [400, 300])
def test_noalloc_matches_regular_entry_point_on_repeated_calls(b):
    """b = 400 (a multiple of 16) runs the tensor-core kernel, b = 300 the
    CUDA-core one; both agree with the regular entry point."""
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    L, Bt, H = 3, 2, 4
    lay, Q = _layout(L, Bt, H, b)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=4, seq_len=b + 32,
                                 budget=b)
    handle = R.reskv_import_cache(cfg, **lay)
    Qd = Q.cuda()
    O_ref = torch.empty(Qd.shape, dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(handle, -1, Qd, O_ref)

    # the same cache in the caller's own device memory
    ks, vs, lc, nm, nr = _device_arrays(lay)
    ref = O_ref.cpu().numpy().astype(np.float64)
    ora = _oracle(lay, Q)
    assert_output_parity(ref, ora, "regular entry point")
    want_kernel = R.RESKV_DECODE_MMA if b % 16 == 0 else R.RESKV_DECODE_FMA
    for call in range(2):
        O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
        R.reskv_decode_attn_noalloc(ks, vs, lc, nm, nr, H, 4, Qd, O)
        assert R.reskv_noalloc_check_status() == want_kernel, f"call {call}"
        out = O.cpu().numpy()
        assert not np.isnan(out).any(), f"call {call}: output not fully written"
        assert_output_parity(out, ref, f"call {call}")
        assert errors(out, ref)[1] < 1e-5, f"call {call}"
        assert_output_parity(out, ora, f"call {call} vs the oracle")
    # per-layer calls through the same scratch
    for l in range(L):
        U_l = Bt * H
        O = torch.empty(Qd[l].shape, dtype=torch.float32, device="cuda")
        sl = slice(l * U_l, (l + 1) * U_l)
        R.reskv_decode_attn_noalloc(ks[sl], vs[sl], lc[sl], nm[sl], nr[sl], H, 4,
                                    Qd[l].contiguous(), O)
        R.reskv_noalloc_check_status()
        assert errors(O.cpu().numpy(), ref[l])[1] < 1e-5
        assert_output_parity(O.cpu().numpy(), ora[l], f"layer {l} vs the oracle")
    handle.free()


def test_noalloc_misaligned_logcounts_take_the_cuda_core_kernel():
    """Log-counts that are not 16-byte aligned rule out the tensor-core
    kernel's bulk copies; the call takes the CUDA-core kernel and still agrees
    with the regular entry point."""
    B.build()
    L, Bt, H, b = 2, 2, 4, 400
    lay, Q = _layout(L, Bt, H, b, seed=11)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=4, seq_len=b + 32,
                                 budget=b)
    handle = R.reskv_import_cache(cfg, **lay)
    Qd = Q.cuda()
    O_ref = torch.empty(Qd.shape, dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(handle, -1, Qd, O_ref)
    U = L * Bt * H
    lc_buf = torch.zeros(U * b + 4, dtype=torch.float32, device="cuda")
    lc = lc_buf[1:1 + U * b].view(U, b)                 # 4 bytes past a 16-byte boundary
    lc.copy_(torch.from_numpy(lay["logc"]).cuda())
    assert lc.data_ptr() % 16 == 4
    ks, vs, lc, nm, nr = _device_arrays(lay, logc=lc)
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn_noalloc(ks, vs, lc, nm, nr, H, 4, Qd, O)
    assert R.reskv_noalloc_check_status() == R.RESKV_DECODE_FMA
    out = O.cpu().numpy()
    ref = O_ref.cpu().numpy().astype(np.float64)
    assert not np.isnan(out).any()
    assert_output_parity(out, ref, "misaligned log-counts")
    assert_output_parity(out, _oracle(lay, Q), "misaligned log-counts vs the oracle")
    assert errors(out, ref)[1] < 1e-5
    handle.free()


def test_noalloc_rejects_calls_beyond_its_scratch():
    """A call whose scratch would exceed the 16 MiB array fails on the host
    with a clear message, before anything is launched."""
    B.build()
    U, b = 65536, 8
    ks = torch.zeros((U, b, 128), dtype=torch.bfloat16, device="cuda")
    lc = torch.zeros((U, b), dtype=torch.float32, device="cuda")
    n = torch.ones(U, dtype=torch.int32, device="cuda")
    Q = torch.zeros((U // 8, 32, 128), dtype=torch.bfloat16, device="cuda")
    O = torch.zeros((U // 8, 32, 128), dtype=torch.float32, device="cuda")
    with pytest.raises(R.ReskvError) as e:
        R.reskv_decode_attn_noalloc(ks, ks, lc, n, n * 0, 8, 4, Q, O)
    assert e.value.status == 2 and "16 MiB" in str(e.value)


@pytest.mark.parametrize("b", [400, 300])
def test_noalloc_status_readback_reports_a_fault_once(b):
    """A bounded wait that gives up (injected: every warp of one call stops at
    its first ring wait) leaves O incomplete; the status readback reports it
    (RESKV_ERR_DEVICE_STATUS, code 1), clears it, and the next call through
    the same scratch is complete and correct."""
    B.build()
    L, Bt, H = 2, 2, 4
    lay, Q = _layout(L, Bt, H, b, seed=5)
    ks, vs, lc, nm, nr = _device_arrays(lay)
    Qd = Q.cuda()
    R.reskv_noalloc_check_status()                      # start from a clear word
    R.reskv_test_inject(R.RESKV_TEST_FAIL_FIRST_WAIT, 1)
    try:
        O = torch.zeros(Qd.shape, dtype=torch.float32, device="cuda")
        R.reskv_decode_attn_noalloc(ks, vs, lc, nm, nr, H, 4, Qd, O)
        with pytest.raises(R.ReskvError) as e:
            R.reskv_noalloc_check_status()
        assert e.value.status == R.RESKV_ERR_DEVICE_STATUS and "word 1" in str(e.value)
        R.reskv_noalloc_check_status()                  # cleared by the read
    finally:
        R.reskv_test_inject(R.RESKV_TEST_FAIL_FIRST_WAIT, 0)
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn_noalloc(ks, vs, lc, nm, nr, H, 4, Qd, O)
    R.reskv_noalloc_check_status()
    assert_output_parity(O.cpu().numpy(), _oracle(lay, Q), "call after the fault")
