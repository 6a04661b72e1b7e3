"""Parity at the workloads' full sizes, in the launch configurations that
bench.py times (one all-layer reskv_decode_attn launch after reskv_build_cache,
and one launch per layer).

The inputs are generated on the GPU by the same generator as the benchmark;
for a seeded sample of units they are regenerated on the CPU (and checked to be
bit-identical), built and decoded by the fp64 oracle, and compared with the
GPU's cache and outputs under the stage-wise protocol of tests/parity.py.
Properties that hold at any size are checked on every unit: per-unit budgets,
the protected window, residual counts, and finite outputs.
"""
import gc

import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import assert_output_parity, bf16_to_f64, errors, unit_from_layout
from parity import check_entries, check_ranking

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


def _units(w, n_sample):
    rng = np.random.default_rng(42)
    if n_sample >= w.n_units:
        return list(range(w.n_units))
    return sorted(int(u) for u in rng.choice(w.n_units, size=n_sample, replace=False))


def run_full(name, n_sample):
    w = wl.WORKLOADS[name]
    L, Bt, H, G = w.n_layers, w.batch, w.n_kv_heads, w.group
    sample = _units(w, n_sample)
    Ks, Vs, Qs = [], [], []
    Qd = torch.empty((L, Bt, H * G, w.head_dim), dtype=torch.bfloat16, device="cuda")
    kept = {}
    for l in range(L):
        K, V, Qo, Qdec = wl.layer_inputs(w, l, "cuda", n_dec_steps=1)
        Ks.append(K)
        Vs.append(V)
        Qs.append(Qo)
        Qd[l] = Qdec[0]
        for u in sample:
            ul, rem = divmod(u, Bt * H)
            if ul == l:
                b, h = divmod(rem, H)
                kept[u] = (K[b, h].cpu(), V[b, h].cpu(),
                           None if Qo is None else Qo[b, h * G:(h + 1) * G].cpu())
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=w.budget, recent_window=w.recent_window, n_obs=w.n_obs,
                                 n_fit=w.n_fit, n_val=w.n_val, score_mode=w.score_mode,
                                 residual_override=w.residual_override(), keep_debug=1)
    cache = R.reskv_build_cache(cfg, Ks, Vs, Qs if w.n_obs > 0 else None)
    del Ks, Vs, Qs
    gc.collect()
    torch.cuda.empty_cache()
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(cache, -1, Qd, O)
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    # one launch per layer (the plan a decode step uses layer by layer)
    O_layers = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    for l in range(L):
        R.reskv_decode_attn(cache, l, Qd[l], O_layers[l])
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    assert errors(O_layers.cpu().numpy(), O.cpu().numpy().astype(np.float64))[1] < 1e-5
    del O_layers
    lay = R.reskv_export_cache(cache)
    scores = R.reskv_export_debug(cache, R.RESKV_DEBUG_SCORES)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED)
    On = O.cpu().numpy()
    qf = bf16_to_f64(Qd)

    # properties of every unit
    P = min(w.recent_window, w.seq_len)
    assert not np.isnan(On).any()
    assert np.all(lay["n_main"] + lay["n_res"] == min(w.budget, w.seq_len))
    assert np.all(lay["n_main"] >= P)
    ovr = w.residual_override()
    if ovr is not None:
        assert np.array_equal(lay["n_res"], ovr)
    for u in range(0, w.n_units, max(1, w.n_units // 64)):
        m, r = lay["n_main"][u], lay["n_res"][u]
        pos = lay["slot_pos"][u, :m]
        assert np.all(np.diff(pos) > 0) and np.all(pos[m - P:] == np.arange(w.seq_len - P, w.seq_len))
        if r > 0:                             # every evicted token sits in one entry
            assert lay["counts"][u, m:m + r].sum() == w.seq_len - m

    # sampled units against the oracle
    swaps, worst = 0, 0.0
    proxy = w.residual == "proxy"
    for u in sample:
        l, rem = divmod(u, Bt * H)
        b, h = divmod(rem, H)
        Kg, Vg, Qg = kept[u]
        Kc, Vc = wl.unit_kv(w, l, b, h, "cpu")
        assert torch.equal(Kc, Kg) and torch.equal(Vc, Vg), "GPU and CPU generators differ"
        Qc = wl.unit_obs_queries(w, l, b, h, Kc, "cpu") if w.n_obs > 0 else None
        if Qc is not None:
            assert torch.equal(Qc, Qg)
        K, V = bf16_to_f64(Kc), bf16_to_f64(Vc)
        Qo = None if Qc is None else bf16_to_f64(Qc)
        oc = orc.OracleConfig(budget=w.budget, recent_window=w.recent_window, n_fit=w.n_fit,
                              n_val=w.n_val, score_mode=w.score_mode,
                              residual_override=None if ovr is None else int(ovr[u]),
                              delta=float(np.float32(cfg.delta)))
        ref = orc.build_unit(K, V, Qo, oc)
        swaps += check_ranking(scores[u], top[u], ref.scores, P, w.score_mode == 1)
        gu = unit_from_layout(lay, u)
        if proxy:
            L_ = ref.losses
            rs = sorted(k for k in L_ if k > 0)
            best = min(rs, key=lambda r: (L_[r], r))
            margin = abs(L_[best] / L_[0] - (1 - oc.delta)) if L_[0] > 0 else 1.0
            vals = sorted(L_[r] for r in rs)
            gap = (vals[1] - vals[0]) / vals[0] if len(vals) > 1 else 1.0
            if min(margin, gap) > 1e-3:
                assert gu.r == ref.r, f"unit {u}: r {gu.r} vs oracle {ref.r}"
        else:
            assert gu.r == ref.r
        check_entries(gu, K, V, top[u], P, w.seq_len, w.budget, 4)
        q = qf[l, b, h * G:(h + 1) * G]
        out = On[l, b, h * G:(h + 1) * G]
        mx, rel = assert_output_parity(out, orc.decode_unit(ref, q, oc), f"unit {u}")
        worst = max(worst, rel)
        own = orc.decode_unit(gu, q, oc)
        assert errors(out, own)[1] < 1e-4, f"unit {u}: kernel vs oracle on the GPU's cache"
    cache.free()
    del O, Qd
    torch.cuda.empty_cache()
    return worst, swaps


def test_llama8b_layer_32k_all_units():
    """One Llama-3.1-8B-shaped layer, s = 32768, b = 512, every unit checked."""
    run_full("llama8b_layer_32k", 8)


def test_llama8b_32l_32k_b8_sampled():
    """The benchmark workload: 32 layers, s = 32768, b = 1024, batch 8."""
    run_full("llama8b_32l_32k_b8", 4)


def test_long_128k_b4_sampled():
    """Long-context stress: 32 layers, s = 131072, b = 2048, batch 4, drift + needles."""
    run_full("long_128k_b4", 2)


def test_small_budget_b64_sampled():
    """Small budget, batch 64: 32 layers, s = 16384, b = 128, key-norm scores, drawn r."""
    run_full("small_budget_b64", 8)
