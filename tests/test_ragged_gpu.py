"""Per-unit (AdaKV-style) budgets through the C ABI: units of different sizes
packed back to back (unit u at sum_{v<u} (b_v + A)), decoded by every decode
path, appended to, and exported, against the fp64 oracle.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import assert_output_parity, bf16_bits, bf16_to_f64, unit_from_layout

pytestmark = pytest.mark.gpu

KERNELS = {"fma": R.RESKV_DECODE_FMA, "mma": R.RESKV_DECODE_MMA,
           "cluster": R.RESKV_DECODE_CLUSTER, "lse": R.RESKV_DECODE_LSE_MERGE,
           "auto": R.RESKV_DECODE_AUTO}


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


def ragged_layout(L, Bt, H, budgets, A, seed=5):
    """Flat layout of units with budgets b_u (+ A append slots each): random
    main/residual splits, some units with unused slots, counts some zero."""
    U = L * Bt * H
    s = int(max(budgets)) + 64
    w = wl.Workload("ragged", L, Bt, H, 4, 128, s, int(max(budgets)), 0, 0, 0, 0, "fixed:0", 1)
    off = np.concatenate([[0], np.cumsum(np.asarray(budgets, np.int64) + A)])
    N = int(off[-1])
    lay = dict(n_main=np.zeros(U, np.int32), n_res=np.zeros(U, np.int32),
               n_app=np.zeros(U, np.int32), kslots=np.zeros((N, 128), np.uint16),
               vslots=np.zeros((N, 128), np.uint16), logc=np.zeros(N, np.float32),
               slot_pos=np.full(N, -1, np.int32), counts=np.zeros(N, np.int32), offsets=off)
    rng = np.random.default_rng(seed)
    for u in range(U):
        bu = int(budgets[u])
        n = bu if u % 3 else int(rng.integers(1, bu + 1))        # every third unit not full
        m = int(rng.integers(1, n + 1))
        r = n - m
        l, rem = divmod(u, Bt * H)
        bb, h = divmod(rem, H)
        K, V = wl.unit_kv(w, l, bb, h)
        o = int(off[u])
        lay["n_main"][u], lay["n_res"][u] = m, r
        lay["kslots"][o:o + n] = bf16_bits(K[:n])
        lay["vslots"][o:o + n] = bf16_bits(V[:n])
        lay["slot_pos"][o:o + m] = np.arange(m)
        if r:
            c = rng.integers(0, 300, r)
            c[rng.random(r) < 0.1] = 0
            lay["counts"][o + m:o + n] = c
            with np.errstate(divide="ignore"):
                lay["logc"][o + m:o + n] = np.log(c.astype(np.float64)).astype(np.float32)
    return w, lay


def import_args(lay):
    return {k: v for k, v in lay.items() if k != "offsets"}


def decode(h, Q, layer=-1):
    Qd = Q.cuda().contiguous()
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(h, layer, Qd, O)
    torch.cuda.synchronize()
    return O.cpu().numpy()


def oracle_outputs(units, Q, L, Bt, H, G):
    qf = bf16_to_f64(Q)
    out = np.zeros(Q.shape)
    oc = orc.OracleConfig(budget=1)
    for l in range(L):
        for bb in range(Bt):
            for h in range(H):
                u = (l * Bt + bb) * H + h
                out[l, bb, h * G:(h + 1) * G] = orc.decode_unit(units[u], qf[l, bb, h * G:(h + 1) * G], oc)
    return out


@pytest.mark.parametrize("kernel", list(KERNELS))
@pytest.mark.parametrize("A", [0, 24])
def test_ragged_budgets_decode_and_append(kernel, A):
    """16 units (2 layers x 2 batch x 4 KV heads) with budgets from 17 to 700
    slots, none a multiple of 16; two rounds of appends when A > 0."""
    L, Bt, H, G = 2, 2, 4, 4
    rng = np.random.default_rng(11)
    budgets = rng.integers(17, 700, L * Bt * H).astype(np.int32)
    budgets[budgets % 16 == 0] += 1
    w, lay = ragged_layout(L, Bt, H, budgets, A)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=int(budgets.mean()), unit_budgets=budgets,
                                 append_capacity=A, decode_kernel=KERNELS[kernel])
    h = R.reskv_import_cache(cfg, **import_args(lay))
    info = R.reskv_get_info(h)
    assert info["ragged"] == 1 and info["total_slots"] == int(lay["offsets"][-1])
    units = [unit_from_layout(lay, u) for u in range(L * Bt * H)]
    g = torch.Generator().manual_seed(13)
    for rnd in range(3 if A else 1):
        if rnd > 0:
            Kn = torch.randn((L, Bt, H, 128), generator=g).to(torch.bfloat16)
            Vn = torch.randn((L, Bt, H, 128), generator=g).to(torch.bfloat16)
            R.reskv_append(h, -1, Kn.cuda(), Vn.cuda())
            kf, vf = bf16_to_f64(Kn), bf16_to_f64(Vn)
            for u in range(L * Bt * H):
                l, rem = divmod(u, Bt * H)
                bb, hh = divmod(rem, H)
                units[u] = orc.append_tokens(units[u], kf[l, bb, hh][None], vf[l, bb, hh][None],
                                             np.array([w.seq_len + rnd - 1]))
        Q = (torch.randn((L, Bt, H * G, 128), generator=g) * 1.5).to(torch.bfloat16)
        ref = oracle_outputs(units, Q, L, Bt, H, G)
        assert_output_parity(decode(h, Q), ref, f"{kernel}, A={A}, round {rnd}, all layers")
        for l in range(L):
            assert_output_parity(decode(h, Q[l], l), ref[l], f"{kernel}, A={A}, round {rnd}, layer {l}")
    R.reskv_check_status(h)
    ex = R.reskv_export_cache(h)
    assert np.array_equal(ex["offsets"], lay["offsets"])
    for u in range(L * Bt * H):
        gu = unit_from_layout(ex, u)
        assert np.array_equal(gu.kmain, units[u].kmain) and np.array_equal(gu.kbar, units[u].kbar)
    h.free()


def test_ragged_budgets_many_units_per_layer():
    """320 units per layer (more than the SMs: stream-K for one-layer calls),
    budgets 1..200, one layer call and the all-layer call."""
    L, Bt, H, G = 2, 40, 8, 4
    rng = np.random.default_rng(17)
    budgets = rng.integers(1, 200, L * Bt * H).astype(np.int32)
    w, lay = ragged_layout(L, Bt, H, budgets, 0, seed=9)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=100, unit_budgets=budgets)
    h = R.reskv_import_cache(cfg, **import_args(lay))
    units = [unit_from_layout(lay, u) for u in range(L * Bt * H)]
    Q = torch.randn((L, Bt, H * G, 128), generator=torch.Generator().manual_seed(2)).to(torch.bfloat16)
    ref = oracle_outputs(units, Q, L, Bt, H, G)
    assert_output_parity(decode(h, Q), ref, "all layers")
    assert_output_parity(decode(h, Q[1], 1), ref[1], "layer 1")
    R.reskv_check_status(h)
