"""GPU construction (Alg. 1) through the C ABI against the fp64 oracle.

Stage-wise protocol (float32 on the GPU, float64 in the oracle):
  scores     relative error <= 1e-4;
  ranking    bit-exact when the oracle ranks the GPU's own scores; against the
             oracle's fp64 scores, two positions may only trade places if their
             fp64 scores differ by < 1e-5 relative (a near tie);
  key-norm   scores and selection bit-exact (both sides give the exact sum of
             the squares rounded once to fp64, in any summation order);
  entries    given the GPU's evicted set in the GPU's rank order, the oracle's
             Lloyd gives the same counts and the same bf16 entries (up to one
             bf16 ulp where the fp32 centres left a near tie);
  r choice   equal unless the oracle's deciding margin is < 1e-3 relative;
  decode     of the GPU-built cache within max abs 1e-2, rel L2 2e-3 of the
             oracle's decode of the oracle-built cache.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import assert_output_parity, bf16_to_f64, errors, unit_from_layout
from parity import (assert_few_skipped, check_entries, check_r, check_ranking, decode_parity,
                    r_margin)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


def make_inputs(w):
    """Inputs drawn on the CPU (the oracle's copies) and uploaded for the library."""
    Ks, Vs, Qs = [], [], []
    for l in range(w.n_layers):
        K, V, Qo, _ = wl.layer_inputs(w, l, "cpu")
        Ks.append(K)
        Vs.append(V)
        Qs.append(Qo)
    up = lambda ts: [None if t is None else t.cuda() for t in ts]
    return (Ks, Vs, Qs), (up(Ks), up(Vs), up(Qs))


def lib_config(w, **kw):
    ovr = w.residual_override()
    return R.reskv_config_default(batch=w.batch, n_layers=w.n_layers, n_kv_heads=w.n_kv_heads,
                                  group=w.group, seq_len=w.seq_len, budget=w.budget,
                                  recent_window=w.recent_window, n_obs=w.n_obs, n_fit=w.n_fit,
                                  n_val=w.n_val, score_mode=w.score_mode,
                                  residual_override=ovr, keep_debug=1, **kw)


def oracle_config(w, cfg):
    ovr = w.residual_override()
    return lambda u: orc.OracleConfig(
        budget=w.budget, recent_window=w.recent_window, n_fit=w.n_fit, n_val=w.n_val,
        score_mode=w.score_mode, residual_override=None if ovr is None else int(ovr[u]),
        delta=float(np.float32(cfg.delta)), gate_mode=cfg.gate_mode, tau=cfg.tau,
        alpha=cfg.alpha, g_min=cfg.g_min, g_fixed=cfg.g_fixed, softmax_mode=cfg.softmax_mode)


def unit_inputs(Ks, Vs, Qs, w, u):
    l, rem = divmod(u, w.batch * w.n_kv_heads)
    b, h = divmod(rem, w.n_kv_heads)
    K = bf16_to_f64(Ks[l][b, h])
    V = bf16_to_f64(Vs[l][b, h])
    Q = None if Qs[l] is None else bf16_to_f64(Qs[l][b, h * w.group:(h + 1) * w.group])
    return K, V, Q


def decode_queries(w, Ks):
    Q = torch.empty((w.n_layers, w.batch, w.n_q_heads, w.head_dim), dtype=torch.bfloat16)
    for l in range(w.n_layers):
        for b in range(w.batch):
            for h in range(w.n_kv_heads):
                k = Ks[l][b, h]
                Q[l, b, h * w.group:(h + 1) * w.group] = \
                    wl.unit_decode_queries(w, l, b, h, k, 1)[:, 0]
    return Q.cuda()


def run_case(w, units=None, **cfg_kw):
    (Ks, Vs, Qs), (Kd, Vd, Qdv) = make_inputs(w)
    cfg = lib_config(w, **cfg_kw)
    Qarg = Qdv if w.n_obs > 0 else None
    cache = R.reskv_build_cache(cfg, Kd, Vd, Qarg)
    R.reskv_check_status(cache)
    # per-stage device times: scores, ranking and packing always run; the
    # validation stages exactly when the proxy decides r
    ms = R.reskv_get_info(cache)["build_ms"]
    proxy_run = w.residual == "proxy" and w.budget < w.seq_len
    assert ms[0] > 0 and ms[1] > 0 and ms[5] > 0
    assert (ms[2] > 0) == proxy_run and (ms[4] > 0) == proxy_run
    lay = R.reskv_export_cache(cache)
    scores = R.reskv_export_debug(cache, R.RESKV_DEBUG_SCORES)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED)
    proxy = w.residual == "proxy" and w.budget < w.seq_len
    P = min(w.recent_window, w.seq_len)
    expect = [r for r in orc.candidate_budgets(w.budget, orc.OracleConfig(budget=1).grid_ratios)
              if w.budget - r >= P] if proxy else []
    cands = R.reskv_export_debug(cache, R.RESKV_DEBUG_CANDIDATES, n_cand=len(expect))
    assert cands.tolist() == expect
    ocfg_of = oracle_config(w, cfg)
    units = range(w.n_units) if units is None else units
    ref_units, swaps, margins = {}, 0, []
    skipped, n_proxy = [], 0
    for u in units:
        K, V, Q = unit_inputs(Ks, Vs, Qs, w, u)
        oc = ocfg_of(u)
        ref = orc.build_unit(K, V, Q, oc)
        ref_units[u] = ref
        swaps += check_ranking(scores[u], top[u], ref.scores, P, w.score_mode == 1)
        gu = unit_from_layout(lay, u)
        if proxy:
            L = ref.losses
            margins.append(r_margin(L, oc.delta))
            n_proxy += 1
            check_r(gu.r, ref, oc.delta, u, skipped)
            gl = R.reskv_export_debug(cache, R.RESKV_DEBUG_LOSSES, n_cand=len(cands))[u]
            np.testing.assert_allclose(gl, [L[0]] + [L[r] for r in cands], rtol=2e-3)
        else:
            assert gu.r == ref.r
        if gu.r == ref.r and set(gu.main_pos.tolist()) != set(ref.main_pos.tolist()):
            # only near-tie swaps may move a token across the boundary
            assert swaps > 0
        check_entries(gu, K, V, top[u], P, w.seq_len, w.budget, 4)
    worst = decode_parity(cache, lay, ref_units, Ks, decode_queries(w, Ks), w, ocfg_of)
    cache.free()
    if n_proxy:
        assert_few_skipped(skipped, n_proxy, w.name)
    return dict(swaps=swaps, worst_rel=worst, margins=margins)


def test_tiny_fixed_residual():
    """Tiny workload: s = 4096, b = 256 with r = 32 fixed, SnapKV scores."""
    out = run_case(wl.WORKLOADS["tiny"])
    assert out["worst_rel"] < 2e-3


def test_proxy_two_heads():
    """Validation proxy (Sec. 5.5.1) on 2 batch x 2 KV heads, s = 2048, b = 256."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=2048, budget=256, batch=2,
                  n_kv_heads=2)
    run_case(w)


def test_proxy_short_window_drift_needles():
    """32-token observation window (24 fit / 8 val) on drifting keys with needles."""
    w = wl.scaled(wl.WORKLOADS["long_128k_b4"], seq_len=4096, budget=512, batch=1, n_layers=2,
                  n_kv_heads=2, n_obs=32, n_fit=24, n_val=8)
    run_case(w)


def test_proxy_separate_softmax_ablation():
    """The "w/o shared softmax" ablation end to end: the validation proxy scores
    candidates and decode mixes the separately normalised branches."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=2048, budget=256, batch=2,
                  n_kv_heads=2)
    out = run_case(w, softmax_mode=R.RESKV_SOFTMAX_SEPARATE)
    assert out["worst_rel"] < 2e-3


def test_keynorm_drawn_residual():
    """Query-free scores, per-(layer, head) drawn r (some 0), s = 2048, b = 128."""
    w = wl.scaled(wl.WORKLOADS["small_budget_b64"], seq_len=2048, batch=3, n_layers=2,
                  n_kv_heads=3)
    run_case(w)


def test_budget_covering_every_token():
    """b >= s: M = S, r = 0, decode = full attention (Eq. attn)."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=600, budget=640, batch=1,
                  n_kv_heads=2)
    out = run_case(w)
    assert out["swaps"] == 0


def _keynorm_rows():
    """Rows (bf16-exact float64 values) where the order or the rounding of the
    sum of squares matters, one per list entry."""
    d = 128
    rows = []
    r = np.full(d, 2.0 ** -13)
    r[0] = 2.0 ** 14                       # in dim order: 2^28; exact: 2^28 + 2^-19
    rows += [r, r[::-1].copy()]
    # a tie at half an ulp of 2^-40 (two squares 2^-94), broken upwards by
    # squares far below the 128-bit window (the wide accumulator) ...
    r = np.full(d, 2.0 ** -126)
    r[:3] = [2.0 ** -20, 2.0 ** -47, 2.0 ** -47]
    rows.append(r)
    # ... by a square inside the window, and not at all (ties to even)
    r = np.zeros(d)
    r[:4] = [2.0 ** -20, 2.0 ** -47, 2.0 ** -47, 2.0 ** -70]
    rows.append(r)
    r = np.zeros(d)
    r[5:8] = [2.0 ** -47, 2.0 ** -20, 2.0 ** -47]
    rows.append(r)
    r = np.zeros(d)                        # bf16 subnormals only
    r[::3] = 2.0 ** -133
    r[1] = 3 * 2.0 ** -130
    rows.append(r)
    rows.append(np.zeros(d))
    r = np.full(d, -(2.0 ** -8))           # signs do not matter
    r[9] = 255 * 2.0 ** -10
    rows.append(r)
    return rows


def test_keynorm_scores_exact_on_crafted_rows():
    """Key-norm scores (a build choice: the exact sum of squares rounded once)
    bit for bit with the oracle on crafted rows and on generator rows, and the
    ranking on them bit-exact; r = 0 so that no other stage sees the rows."""
    s, b, P = 1024, 256, 64
    w = wl.scaled(wl.WORKLOADS["small_budget_b64"], seq_len=s, budget=b, batch=1, n_layers=1,
                  n_kv_heads=2)
    K, V, _, _ = wl.layer_inputs(w, 0, "cpu")
    rows = _keynorm_rows()
    for h in range(2):
        for i, row in enumerate(rows):
            t = torch.from_numpy(row.astype(np.float32)).to(torch.bfloat16)
            assert np.array_equal(t.double().numpy(), row)          # exact in bf16
            K[0, h, 100 * h + 37 * i] = t
    cfg = R.reskv_config_default(batch=1, n_layers=1, n_kv_heads=2, group=w.group, seq_len=s,
                                 budget=b, recent_window=P, n_obs=0, n_fit=0, n_val=0,
                                 score_mode=R.RESKV_SCORE_KEYNORM,
                                 residual_override=np.zeros(2, np.int32), keep_debug=1)
    cache = R.reskv_build_cache(cfg, [K.cuda()], [V.cuda()], None)
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    scores = R.reskv_export_debug(cache, R.RESKV_DEBUG_SCORES).reshape(2, s)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED).reshape(2, -1)
    for h in range(2):
        Kf = K[0, h].double().numpy()
        ref = orc.scores_keynorm(Kf)
        bad = np.nonzero(scores[h] != ref)[0]
        assert bad.size == 0, (h, bad[:5], scores[h][bad[:5]], ref[bad[:5]])
        check_ranking(scores[h], top[h], ref, P, keynorm=True)
    p0 = 37 * 0
    assert scores[0][p0] == 2.0 ** 28 + 2.0 ** -19
    assert scores[0][37 * 2] == 2.0 ** -40 + 2.0 ** -92
    assert scores[0][37 * 3] == 2.0 ** -40 + 2.0 ** -92
    assert scores[0][37 * 4] == 2.0 ** -40
    assert scores[0][37 * 6] == 0.0
    cache.free()


def test_lloyd_sums_outside_the_fixed_point_range():
    """Centre means (Eq. summary) when member values leave the exact
    fixed-point range of the member sums (multiples of 2^-32 below 128): every
    key carries a dim of values 2^-40 m (m up to 255), some keys a bf16
    subnormal, and some values 2^40.  Those centres take the fp64 member-order
    sums; counts and bf16 entries must match the oracle's Lloyd on the same
    evicted set, and a missed range check (a truncated or saturated sum) would
    not."""
    s, b, P, r = 1024, 256, 64, 8
    w = wl.scaled(wl.WORKLOADS["small_budget_b64"], seq_len=s, budget=b, batch=1, n_layers=1,
                  n_kv_heads=2)
    K, V, _, _ = wl.layer_inputs(w, 0, "cpu")
    g = np.random.default_rng(7)
    for h in range(2):
        m = g.integers(1, 256, size=s) * g.choice([-1.0, 1.0], size=s)
        K[0, h, :, 5] = torch.from_numpy(m * 2.0 ** -40).to(torch.bfloat16)
        K[0, h, ::97, 9] = 2.0 ** -133
        V[0, h, 3::41, 7] = 2.0 ** 40
        assert torch.all(K[0, h, :, 5].double() == torch.from_numpy(m * 2.0 ** -40))
    cfg = R.reskv_config_default(batch=1, n_layers=1, n_kv_heads=2, group=w.group, seq_len=s,
                                 budget=b, recent_window=P, n_obs=0, n_fit=0, n_val=0,
                                 score_mode=R.RESKV_SCORE_KEYNORM,
                                 residual_override=np.full(2, r, np.int32), keep_debug=1)
    cache = R.reskv_build_cache(cfg, [K.cuda()], [V.cuda()], None)
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    lay = R.reskv_export_cache(cache)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED)
    big = 0
    for h in range(2):
        gu = unit_from_layout(lay, h)
        assert gu.r == r
        check_entries(gu, bf16_to_f64(K[0, h]), bf16_to_f64(V[0, h]), top[h], P, s, b, 4)
        big += int(np.sum(np.abs(gu.vbar[:, 7]) > 2.0 ** 20))
    assert big > 0                       # some centre holds a 2^40 value
    cache.free()


def test_lloyd_at_the_persistent_assignment_edges():
    """Lloyd (Sec. 5.3) with r at the edges of the persistent assignment:
    r = 1 (one centre among padded keys), 16 and 17 (one and two 16-column
    MMA blocks), 255 and 256 (the most centres held in shared memory), and
    r = 0 units between them, in one layer; in the other layer 257 and 300
    switch that layer's runs to the streaming form.  Counts bit-exact and
    entries within one bf16 ulp of the oracle's Lloyd on the GPU's evicted
    set, for every unit."""
    s, b, P = 2048, 512, 64
    w = wl.scaled(wl.WORKLOADS["small_budget_b64"], seq_len=s, budget=b, batch=4, n_layers=2,
                  n_kv_heads=2)
    ovr = np.array([1, 16, 17, 0, 255, 256, 0, 40,            # layer 0: persistent
                    257, 300, 0, 33, 1, 256, 128, 2], np.int32)  # layer 1: streaming
    assert ovr.size == w.n_units
    Ks, Vs = [], []
    for l in range(w.n_layers):
        K, V, _, _ = wl.layer_inputs(w, l, "cpu")
        Ks.append(K)
        Vs.append(V)
    cfg = R.reskv_config_default(batch=w.batch, n_layers=w.n_layers, n_kv_heads=w.n_kv_heads,
                                 group=w.group, seq_len=s, budget=b, recent_window=P, n_obs=0,
                                 n_fit=0, n_val=0, score_mode=R.RESKV_SCORE_KEYNORM,
                                 residual_override=ovr, keep_debug=1)
    cache = R.reskv_build_cache(cfg, [k.cuda() for k in Ks], [v.cuda() for v in Vs], None)
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    lay = R.reskv_export_cache(cache)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED)
    for u in range(w.n_units):
        l, rem = divmod(u, w.batch * w.n_kv_heads)
        bb, h = divmod(rem, w.n_kv_heads)
        gu = unit_from_layout(lay, u)
        assert gu.r == ovr[u], (u, gu.r, ovr[u])
        check_entries(gu, bf16_to_f64(Ks[l][bb, h]), bf16_to_f64(Vs[l][bb, h]), top[u], P, s, b, 4)
    cache.free()
