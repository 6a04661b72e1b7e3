"""Decode-time append (Sec. 3.1: each decode step appends the new token's key
and value) through the C ABI: rows added with reskv_append join the exact main
cache of their unit, and every decode path attends to them.  The reference is
the fp64 oracle's append_tokens on the same rows.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import (assert_output_parity, bf16_bits, bf16_to_f64, errors, unit_from_layout)
from test_build_gpu import lib_config, make_inputs
from test_decode_gpu import SPLITS, synthetic_layout

pytestmark = pytest.mark.gpu

KERNELS = {"fma": R.RESKV_DECODE_FMA, "mma": R.RESKV_DECODE_MMA,
           "cluster": R.RESKV_DECODE_CLUSTER, "lse": R.RESKV_DECODE_LSE_MERGE,
           "auto": R.RESKV_DECODE_AUTO}


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


def with_capacity(lay: dict, A: int) -> dict:
    """The same units with A more slots per unit (unit stride b + A)."""
    out = {}
    for k, v in lay.items():
        if v.ndim >= 2:
            pad = [(0, 0), (0, A)] + [(0, 0)] * (v.ndim - 2)
            out[k] = np.pad(v, pad, constant_values=-1 if k == "slot_pos" else 0)
        else:
            out[k] = v.copy()
    out["n_app"] = np.zeros(len(lay["n_main"]), np.int32)
    return out


def oracle_outputs(units, Q, L, Bt, H, G, ocfg):
    qf = bf16_to_f64(Q)
    out = np.zeros(Q.shape)
    for l in range(L):
        for bb in range(Bt):
            for h in range(H):
                u = (l * Bt + bb) * H + h
                out[l, bb, h * G:(h + 1) * G] = orc.decode_unit(units[u], qf[l, bb, h * G:(h + 1) * G],
                                                                ocfg)
    return out


def decode(h, Q, layer=-1):
    Qd = Q.cuda().contiguous()
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(h, layer, Qd, O)
    torch.cuda.synchronize()
    return O.cpu().numpy()


@pytest.mark.parametrize("kernel", list(KERNELS))
def test_appended_tokens_join_the_main_cache(kernel):
    """12 ragged units (b = 300, room for 40 appended rows each); five rounds
    of appends, per layer and for all layers at once, each followed by
    all-layer and per-layer decodes whose queries favour the newest rows."""
    L, Bt, H, G, b, A = 2, 3, 2, 4, 300, 40
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    lay = with_capacity(lay, A)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b, append_capacity=A, decode_kernel=KERNELS[kernel])
    h = R.reskv_import_cache(cfg, **lay)
    ocfg = orc.OracleConfig(budget=b)
    units = [unit_from_layout(lay, u) for u in range(L * Bt * H)]
    g = torch.Generator().manual_seed(7)
    rounds = 5
    for step in range(rounds):
        Kn = torch.randn((L, Bt, H, 128), generator=g).to(torch.bfloat16)
        Vn = (3.0 * torch.randn((L, Bt, H, 128), generator=g)).to(torch.bfloat16)
        if step % 2 == 0:
            for l in range(L):
                R.reskv_append(h, l, Kn[l].cuda(), Vn[l].cuda())
        else:
            R.reskv_append(h, -1, Kn.cuda(), Vn.cuda())
        kf, vf = bf16_to_f64(Kn), bf16_to_f64(Vn)
        for l in range(L):
            for bb in range(Bt):
                for hh in range(H):
                    u = (l * Bt + bb) * H + hh
                    units[u] = orc.append_tokens(units[u], kf[l, bb, hh][None], vf[l, bb, hh][None],
                                                 np.array([w.seq_len + step]))
        # queries: half the heads aim at the newest row (0.7 k_new + noise)
        Q = torch.randn((L, Bt, H * G, 128), generator=g)
        for gg in range(0, G, 2):
            Q[:, :, gg::G] = 2.0 * Kn.float() + 0.3 * Q[:, :, gg::G]
        Q = Q.to(torch.bfloat16)
        ref = oracle_outputs(units, Q, L, Bt, H, G, ocfg)
        assert_output_parity(decode(h, Q), ref, f"{kernel}, round {step}, all layers")
        for l in range(L):
            assert_output_parity(decode(h, Q[l], l), ref[l], f"{kernel}, round {step}, layer {l}")
    R.reskv_check_status(h)
    info = R.reskv_get_info(h)
    assert (info["append_capacity"], info["stride"], info["max_appended"]) == (A, b + A, rounds)
    ex = R.reskv_export_cache(h)
    assert np.all(ex["n_app"] == rounds)
    assert np.array_equal(ex["n_main"], lay["n_main"]) and np.array_equal(ex["n_res"], lay["n_res"])
    for u in range(L * Bt * H):
        m, r = int(lay["n_main"][u]), int(lay["n_res"][u])
        assert ex["slot_pos"][u, m + r:m + r + rounds].tolist() == [w.seq_len + i for i in range(rounds)]
        gu = unit_from_layout(ex, u)
        assert np.array_equal(gu.kmain, units[u].kmain) and np.array_equal(gu.vmain, units[u].vmain)
    h.free()


def test_append_region_full_is_rejected_without_writing():
    L, Bt, H, b, A = 1, 2, 2, 64, 3
    w, lay = synthetic_layout(L, Bt, H, b, [(60, 4), (64, 0), (10, 20), (33, 1)])
    lay = with_capacity(lay, A)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=4, seq_len=w.seq_len,
                                 budget=b, append_capacity=A)
    h = R.reskv_import_cache(cfg, **lay)
    Kn = torch.ones((Bt, H, 128), dtype=torch.bfloat16, device="cuda")
    for _ in range(A):
        R.reskv_append(h, 0, Kn, Kn)
    with pytest.raises(R.ReskvError) as e:
        R.reskv_append(h, 0, Kn, Kn)
    assert e.value.status == R.RESKV_ERR_UNSUPPORTED and "full" in str(e.value)
    assert np.all(R.reskv_export_cache(h)["n_app"] == A)
    R.reskv_check_status(h)
    # a cache without append capacity rejects the first append
    cfg0 = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=4, seq_len=w.seq_len,
                                  budget=b)
    lay0 = {k: v[:, :b] if v.ndim >= 2 else v for k, v in lay.items() if k != "n_app"}
    h0 = R.reskv_import_cache(cfg0, **lay0)
    with pytest.raises(R.ReskvError):
        R.reskv_append(h0, 0, Kn, Kn)


def test_build_with_append_capacity_packs_the_same_cache():
    """reskv_build_cache with room for appends lays out the same units at the
    wider stride, and decodes the same outputs."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=2048, budget=256, batch=2,
                  n_kv_heads=2)
    (Ks, Vs, Qs), (Kd, Vd, Qdv) = make_inputs(w)
    c0 = R.reskv_build_cache(lib_config(w), Kd, Vd, Qdv)
    c1 = R.reskv_build_cache(lib_config(w, append_capacity=24), Kd, Vd, Qdv)
    e0, e1 = R.reskv_export_cache(c0), R.reskv_export_cache(c1)
    for k in ("n_main", "n_res"):
        assert np.array_equal(e0[k], e1[k])
    for k in ("kslots", "vslots", "logc", "slot_pos", "counts"):
        assert np.array_equal(e0[k], e1[k][:, :w.budget]), k
    assert np.all(e1["slot_pos"][:, w.budget:] == -1) and np.all(e1["n_app"] == 0)
    Q = torch.randn((w.n_layers, w.batch, w.n_kv_heads * w.group, 128),
                    generator=torch.Generator().manual_seed(3)).to(torch.bfloat16)
    o0, o1 = decode(c0, Q), decode(c1, Q)
    assert errors(o1, o0.astype(np.float64))[1] < 1e-5
