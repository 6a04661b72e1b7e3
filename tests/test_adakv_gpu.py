"""Construction with per-unit budgets through the C ABI against the fp64 oracle:
AdaKV's allocation across KV heads (App. B, "AdaKV"; the "+ResKV" rows of
Table ruler_paper and Table longbench_paper) and caller-given budgets, each
unit then built by Alg. 1 with its own budget.

Protocol (float32 scores on the GPU, float64 in the oracle):
  budgets    bit-exact when the oracle allocates from the GPU's own scores;
             against the oracle's fp64 scores equal unless the pooled pick's
             boundary is a near tie (< 1e-5 relative); key-norm scores are
             exact on both sides, so their budgets are bit-exact outright;
  per unit   the stage-wise protocol of the uniform-budget construction
             (ranking, entries, r choice) with the unit's budget, and the
             decode of the built cache within max abs 1e-2, rel L2 2e-3.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import assert_output_parity, bf16_to_f64, unit_from_layout
from parity import NEAR_TIE, assert_few_skipped, check_entries, check_r, check_ranking

pytestmark = pytest.mark.gpu

SAFEGUARD = 0.2
KERNELS = {"fma": R.RESKV_DECODE_FMA, "mma": R.RESKV_DECODE_MMA,
           "cluster": R.RESKV_DECODE_CLUSTER, "lse": R.RESKV_DECODE_LSE_MERGE,
           "auto": R.RESKV_DECODE_AUTO}


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


def make_inputs(w, sharpen_head=None):
    """CPU inputs (the oracle's copies) and their device uploads.  Keys of
    `sharpen_head` are doubled (exact in bf16) so that its attention is
    sharper and the allocation moves budget towards or away from it."""
    Ks, Vs, Qs = [], [], []
    for l in range(w.n_layers):
        K, V, Qo, _ = wl.layer_inputs(w, l, "cpu")
        if sharpen_head is not None:
            K[:, sharpen_head] *= 2
        Ks.append(K)
        Vs.append(V)
        Qs.append(Qo)
    up = lambda ts: [None if t is None else t.cuda() for t in ts]
    return (Ks, Vs, Qs), (up(Ks), up(Vs), up(Qs))


def lib_config(w, **kw):
    return R.reskv_config_default(batch=w.batch, n_layers=w.n_layers, n_kv_heads=w.n_kv_heads,
                                  group=w.group, seq_len=w.seq_len, budget=w.budget,
                                  recent_window=w.recent_window, n_obs=w.n_obs, n_fit=w.n_fit,
                                  n_val=w.n_val, score_mode=w.score_mode,
                                  residual_override=w.residual_override(), keep_debug=1, **kw)


def oracle_config(w, cfg, budget, u):
    ovr = w.residual_override()
    return orc.OracleConfig(
        budget=int(budget), recent_window=w.recent_window, n_fit=w.n_fit, n_val=w.n_val,
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
                Q[l, b, h * w.group:(h + 1) * w.group] = \
                    wl.unit_decode_queries(w, l, b, h, Ks[l][b, h], 1)[:, 0]
    return Q


def pooled_gap(scores, budget, recent, safeguard):
    """Relative gap between the last pooled pick and the first token left out
    (the near-tie margin of the AdaKV allocation)."""
    H, s = scores.shape
    n_p = min(recent, s)
    n = budget - n_p
    f = int(np.floor(float(np.float32(safeguard)) * n))
    pool = np.sort(np.concatenate([scores[h][orc.rank_evictable(scores[h], recent)[f:]]
                                   for h in range(H)]))[::-1]
    k = H * (n - f)
    if k == 0 or k >= len(pool):
        return 1.0
    a, b = pool[k - 1], pool[k]
    return abs(a - b) / max(abs(a), abs(b), 1e-300)


def check_budgets(w, gpu_budgets, gpu_scores, ref_scores, exact):
    """Budget protocol per (layer, batch element); returns the number of groups
    whose oracle allocation differs at a near tie."""
    H, P = w.n_kv_heads, min(w.recent_window, w.seq_len)
    n = w.budget - P
    f = int(np.floor(float(np.float32(SAFEGUARD)) * n))
    near = 0
    for g in range(w.n_layers * w.batch):
        sl = slice(g * H, (g + 1) * H)
        got = gpu_budgets[sl]
        assert got.sum() == H * w.budget and np.all(got >= P + f) and np.all(got <= w.seq_len)
        own = orc.adakv_budgets(gpu_scores[sl], w.budget, w.recent_window, SAFEGUARD)
        assert np.array_equal(own, got), f"group {g}: GPU budgets differ from its own scores'"
        ref = orc.adakv_budgets(ref_scores[sl], w.budget, w.recent_window, SAFEGUARD)
        if not np.array_equal(ref, got):
            assert not exact, f"group {g}: exact scores but budgets {got} vs oracle {ref}"
            assert pooled_gap(ref_scores[sl], w.budget, w.recent_window, SAFEGUARD) < NEAR_TIE
            near += 1
    return near


def run_per_unit(w, budgets_in=None, sharpen_head=None, **cfg_kw):
    """Build with AdaKV (budgets_in None) or the given per-unit budgets; check
    every unit stage-wise against the oracle built with its budget, then the
    decode of the whole cache."""
    (Ks, Vs, Qs), (Kd, Vd, Qdv) = make_inputs(w, sharpen_head)
    if budgets_in is None:
        cfg = lib_config(w, budget_mode=R.RESKV_BUDGET_ADAKV, adakv_safeguard=SAFEGUARD, **cfg_kw)
    else:
        cfg = lib_config(w, unit_budgets=budgets_in, **cfg_kw)
    cache = R.reskv_build_cache(cfg, Kd, Vd, Qdv if w.n_obs > 0 else None)
    R.reskv_check_status(cache)
    info = R.reskv_get_info(cache)
    budgets = R.reskv_get_unit_budgets(cache)
    scores = R.reskv_export_debug(cache, R.RESKV_DEBUG_SCORES)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED)
    lay = R.reskv_export_cache(cache)
    P = min(w.recent_window, w.seq_len)
    keynorm = w.score_mode == 1
    proxy = w.residual == "proxy"
    refs = {}
    ref_scores = np.zeros_like(scores)
    for u in range(w.n_units):
        K, V, Q = unit_inputs(Ks, Vs, Qs, w, u)
        ref_scores[u] = orc.unit_scores(K, Q, oracle_config(w, cfg, w.budget, u))
    near = 0
    if budgets_in is None:
        assert info["ragged"] == 1 and info["total_slots"] == w.n_units * w.budget
        near = check_budgets(w, budgets, scores, ref_scores, keynorm)
    else:
        assert np.array_equal(budgets, budgets_in)
    if proxy:
        ucands = R.reskv_export_debug(cache, R.RESKV_DEBUG_UNIT_CANDIDATES)
        losses = R.reskv_export_debug(cache, R.RESKV_DEBUG_LOSSES)
        ratios = sorted({float(np.float32(x)) for x in orc.OracleConfig(budget=1).grid_ratios
                         if x > 0})
    swaps = 0
    skipped, n_proxy = [], 0
    for u in range(w.n_units):
        K, V, Q = unit_inputs(Ks, Vs, Qs, w, u)
        bu = int(budgets[u])
        oc = oracle_config(w, cfg, bu, u)
        ref = orc.build_unit(K, V, Q, oc)
        refs[u] = ref
        width = max(min(bu, w.seq_len) - P, 0)
        assert np.all(top[u, width:] == -1)
        swaps += check_ranking(scores[u], top[u, :width], ref.scores, P, keynorm)
        gu = unit_from_layout(lay, u)
        assert len(gu.main_pos) + gu.r <= bu
        if proxy and bu < w.seq_len:
            # the unit's candidate columns: floor(ratio * b_u), valid and distinct
            expect = [r for r in orc.candidate_budgets(bu, orc.OracleConfig(budget=1).grid_ratios)
                      if orc.candidate_valid(w.seq_len, oc, r)]
            cols = [r for r in ucands[u] if r > 0]
            assert cols == expect, f"unit {u}: candidates {cols} vs oracle {expect}"
            assert all(r == 0 or int(np.floor(ratios[i] * bu)) == r
                       for i, r in enumerate(ucands[u]))
            L = ref.losses
            np.testing.assert_allclose(losses[u, 0], L[0], rtol=2e-3)
            for i, r in enumerate(ucands[u]):
                if r > 0:
                    np.testing.assert_allclose(losses[u, 1 + i], L[r], rtol=2e-3)
                else:
                    assert losses[u, 1 + i] == np.inf
            rs = sorted(k for k in L if k > 0)
            if rs:
                n_proxy += 1
                check_r(gu.r, ref, oc.delta, u, skipped)
            else:
                assert gu.r == 0
        else:
            assert gu.r == ref.r
        if gu.r == ref.r and set(gu.main_pos.tolist()) != set(ref.main_pos.tolist()):
            assert swaps > 0
        check_entries(gu, K, V, top[u, :width], P, w.seq_len, bu, 4)
    # decode of the built cache (automatic plan) against the oracle's caches
    Qd = decode_queries(w, Ks)
    out = decode_all(cache, Qd.cuda())
    worst = compare_decode(out, Qd, refs, lay, w, lambda u: oracle_config(w, cfg, budgets[u], u))
    cache.free()
    if n_proxy:
        assert_few_skipped(skipped, n_proxy, w.name)
    return dict(budgets=budgets, near=near, swaps=swaps, worst=worst, lay=lay, refs=refs,
                Ks=Ks, cfg=cfg)


def decode_all(cache, Qd):
    O = torch.empty(Qd.shape, dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(cache, -1, Qd, O)
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    return O.cpu().numpy()


def compare_decode(O, Qd, refs, lay, w, ocfg_of):
    qf = bf16_to_f64(Qd)
    G, H, Bt = w.group, w.n_kv_heads, w.batch
    worst = 0.0
    for u, ref in refs.items():
        l, rem = divmod(u, Bt * H)
        b, h = divmod(rem, H)
        q = qf[l, b, h * G:(h + 1) * G]
        got = O[l, b, h * G:(h + 1) * G]
        _, rel = assert_output_parity(got, orc.decode_unit(ref, q, ocfg_of(u)), f"unit {u}")
        own = orc.decode_unit(unit_from_layout(lay, u), q, ocfg_of(u))
        assert_output_parity(got, own, f"unit {u} (own cache)")
        worst = max(worst, rel)
    return worst


def test_adakv_proxy_snapkv_scores():
    """AdaKV with SnapKV scores and the validation proxy per head: 2 layers x
    2 batch x 4 KV heads, s = 2048, b = 256, one head's keys doubled."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=2048, budget=256, batch=2,
                  n_kv_heads=4, n_layers=2)
    out = run_per_unit(w, sharpen_head=1)
    b = out["budgets"]
    assert len(set(b.tolist())) > 4, f"allocation is not ragged: {b}"
    assert out["worst"] < 2e-3


def test_adakv_keynorm_fixed_residual_bit_exact_budgets():
    """Query-free key-norm scores (exact on both sides): the budgets must equal
    the oracle's outright; r per (layer, head) drawn, some 0."""
    # the smallest AdaKV budget, |P| + floor(0.2 (b - |P|)) = 128, leaves room
    # for |P| = 64 main slots beside the largest drawn r (64)
    w = wl.scaled(wl.WORKLOADS["small_budget_b64"], seq_len=2048, budget=384, batch=2,
                  n_layers=2, n_kv_heads=4)
    out = run_per_unit(w, sharpen_head=2)
    assert out["near"] == 0
    # head 2's doubled keys outscore every other head's: it takes every shared
    # slot, b_2 = |P| + f + H (b - |P| - f) = 64 + 64 + 4 * 256
    b = out["budgets"].reshape(-1, w.n_kv_heads)
    assert np.all(b[:, 2] == 1152) and np.all(np.delete(b, 2, axis=1) == 128)


def test_adakv_drift_needles_short_window():
    """Drifting keys with needles, 32-token observation window (24 fit / 8 val)."""
    w = wl.scaled(wl.WORKLOADS["long_128k_b4"], seq_len=4096, budget=384, batch=1, n_layers=2,
                  n_kv_heads=4, n_obs=32, n_fit=24, n_val=8)
    run_per_unit(w, sharpen_head=0)


def test_caller_budgets_with_the_proxy():
    """Per-unit budgets given by the caller (two of them cover every token):
    the proxy's candidates follow each unit's budget."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=1024, budget=256, batch=2,
                  n_kv_heads=3, n_layers=2)
    rng = np.random.default_rng(11)
    budgets = rng.integers(70, 600, w.n_units).astype(np.int32)
    budgets[3], budgets[7] = 1024, 1500
    out = run_per_unit(w, budgets_in=budgets)
    assert out["worst"] < 2e-3


def test_adakv_with_budget_covering_every_token_stays_uniform():
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=300, budget=320, batch=1,
                  n_kv_heads=2)
    (Ks, Vs, Qs), (Kd, Vd, Qdv) = make_inputs(w)
    cfg = lib_config(w, budget_mode=R.RESKV_BUDGET_ADAKV)
    cache = R.reskv_build_cache(cfg, Kd, Vd, Qdv)
    info = R.reskv_get_info(cache)
    assert info["ragged"] == 0
    assert R.reskv_get_unit_budgets(cache).tolist() == [320, 320]
    lay = R.reskv_export_cache(cache)
    assert lay["n_main"].tolist() == [300, 300] and lay["n_res"].tolist() == [0, 0]
    cache.free()


def test_adakv_rejects_caller_budgets_and_bad_safeguard():
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=512, budget=128, batch=1,
                  n_kv_heads=2)
    (_, _, _), (Kd, Vd, Qdv) = make_inputs(w)
    for kw in (dict(budget_mode=R.RESKV_BUDGET_ADAKV, unit_budgets=np.array([128, 128], np.int32)),
               dict(budget_mode=R.RESKV_BUDGET_ADAKV, adakv_safeguard=1.5),
               dict(budget_mode=7)):
        with pytest.raises(R.ReskvError) as e:
            R.reskv_build_cache(lib_config(w, **kw), Kd, Vd, Qdv)
        assert e.value.status == R.RESKV_ERR_INVALID_ARG


@pytest.mark.parametrize("kernel", sorted(KERNELS))
def test_adakv_cache_on_every_decode_path(kernel):
    """The AdaKV-built cache, exported and imported with its budgets, decoded
    by every decode path, per layer and all layers."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=1024, budget=160, batch=2,
                  n_kv_heads=4, n_layers=2)
    (Ks, Vs, Qs), (Kd, Vd, Qdv) = make_inputs(w, sharpen_head=3)
    cfg = lib_config(w, budget_mode=R.RESKV_BUDGET_ADAKV)
    built = R.reskv_build_cache(cfg, Kd, Vd, Qdv)
    budgets = R.reskv_get_unit_budgets(built)
    lay = R.reskv_export_cache(built)
    built.free()
    icfg = lib_config(w, unit_budgets=budgets, decode_kernel=KERNELS[kernel])
    cache = R.reskv_import_cache(icfg, lay["n_main"], lay["n_res"], lay["kslots"], lay["vslots"],
                                 lay["logc"], lay["slot_pos"], lay["counts"])
    Qd = decode_queries(w, Ks)
    ocfg = lambda u: oracle_config(w, cfg, budgets[u], u)
    refs = {u: unit_from_layout(lay, u) for u in range(w.n_units)}
    compare_decode(decode_all(cache, Qd.cuda()), Qd, refs, lay, w, ocfg)
    O = np.zeros((w.n_layers,) + tuple(Qd.shape[1:]), np.float32)
    for l in range(w.n_layers):
        Ol = torch.empty(Qd.shape[1:], dtype=torch.float32, device="cuda")
        R.reskv_decode_attn(cache, l, Qd[l].cuda().contiguous(), Ol)
        torch.cuda.synchronize()
        O[l] = Ol.cpu().numpy()
    R.reskv_check_status(cache)
    compare_decode(O, Qd, refs, lay, w, ocfg)
    cache.free()


def test_adakv_fullsize_bench_workload_sampled():
    """The benchmark workload (32 layers, s = 32768, b = 1024, batch 8) built
    with AdaKV budgets, decoded in the launch configurations bench.py times.
    Every (layer, batch element) keeps 8 x 1024 slots; two sampled groups'
    allocations against the oracle; one unit of each against the oracle built
    with its budget."""
    import gc
    w = wl.WORKLOADS["llama8b_32l_32k_b8"]
    L, Bt, H, G = w.n_layers, w.batch, w.n_kv_heads, w.group
    groups = [(3, 5), (27, 1)]                      # (layer, batch element)
    Ks, Vs, Qs, kept = [], [], [], {}
    Qd = torch.empty((L, Bt, H * G, w.head_dim), dtype=torch.bfloat16, device="cuda")
    for l in range(L):
        K, V, Qo, Qdec = wl.layer_inputs(w, l, "cuda", n_dec_steps=1)
        Ks.append(K)
        Vs.append(V)
        Qs.append(Qo)
        Qd[l] = Qdec[0]
        for (gl, gb) in groups:
            if gl == l:
                kept[(gl, gb)] = (K[gb].cpu(), V[gb].cpu(), Qo[gb].cpu())
    cfg = lib_config(w, budget_mode=R.RESKV_BUDGET_ADAKV)
    cache = R.reskv_build_cache(cfg, Ks, Vs, Qs)
    del Ks, Vs, Qs
    gc.collect()
    torch.cuda.empty_cache()
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(cache, -1, Qd, O)
    O_layers = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    for l in range(L):
        R.reskv_decode_attn(cache, l, Qd[l], O_layers[l])
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    On = O.cpu().numpy()
    assert not np.isnan(On).any()
    assert np.abs(O_layers.cpu().numpy() - On).max() <= 1e-5 * max(1.0, np.abs(On).max())
    budgets = R.reskv_get_unit_budgets(cache)
    P = w.recent_window
    f = int(np.floor(float(np.float32(SAFEGUARD)) * (w.budget - P)))
    bg = budgets.reshape(L * Bt, H)
    assert np.all(bg.sum(axis=1) == H * w.budget) and np.all(bg >= P + f)
    assert len(np.unique(bg)) > 16, "the allocation is not ragged"
    info = R.reskv_get_info(cache)
    assert info["ragged"] == 1 and info["total_slots"] == w.n_units * w.budget
    lay = R.reskv_export_cache(cache)
    assert np.all(lay["n_main"] + lay["n_res"] == budgets)
    scores = R.reskv_export_debug(cache, R.RESKV_DEBUG_SCORES)
    top = R.reskv_export_debug(cache, R.RESKV_DEBUG_RANKED)
    qf = bf16_to_f64(Qd)
    skipped_full, n_full = [], 0
    for (gl, gb) in groups:
        Kg, Vg, Qg = kept[(gl, gb)]
        u0 = (gl * Bt + gb) * H
        sl = slice(u0, u0 + H)
        ref_scores = np.stack([orc.unit_scores(bf16_to_f64(Kg[h]), bf16_to_f64(Qg[h * G:(h + 1) * G]),
                                               oracle_config(w, cfg, w.budget, u0 + h))
                               for h in range(H)])
        own = orc.adakv_budgets(scores[sl], w.budget, P, SAFEGUARD)
        assert np.array_equal(own, budgets[sl]), f"group {(gl, gb)}: budgets vs its own scores"
        ref = orc.adakv_budgets(ref_scores, w.budget, P, SAFEGUARD)
        if not np.array_equal(ref, budgets[sl]):
            assert pooled_gap(ref_scores, w.budget, P, SAFEGUARD) < NEAR_TIE
        h = int(np.argmax(budgets[sl]))              # the head with the largest budget
        u = u0 + h
        bu = int(budgets[u])
        K, V, Q = bf16_to_f64(Kg[h]), bf16_to_f64(Vg[h]), bf16_to_f64(Qg[h * G:(h + 1) * G])
        oc = oracle_config(w, cfg, bu, u)
        refu = orc.build_unit(K, V, Q, oc)
        width = bu - P
        check_ranking(scores[u], top[u, :width], refu.scores, P, False)
        gu = unit_from_layout(lay, u)
        check_r(gu.r, refu, oc.delta, u, skipped_full)
        n_full += 1
        check_entries(gu, K, V, top[u, :width], P, w.seq_len, bu, 4)
        q = qf[gl, gb, h * G:(h + 1) * G]
        out = On[gl, gb, h * G:(h + 1) * G]
        assert_output_parity(out, orc.decode_unit(refu, q, oc), f"unit {u}")
        assert_output_parity(out, orc.decode_unit(gu, q, oc), f"unit {u} (own cache)")
    assert_few_skipped(skipped_full, n_full, "adakv full size")
    cache.free()
    del O, O_layers, Qd
    torch.cuda.empty_cache()


@pytest.mark.parametrize("group", [2, 4])
def test_adakv_build_then_append(group):
    """AdaKV construction at the wider unit stride (append capacity 6), then
    three rounds of appended tokens: every unit's exact main cache grows
    inside its own region and decodes (all-layer and per-layer) against the
    oracle's cache grown by append_tokens."""
    w = wl.scaled(wl.WORKLOADS["llama8b_layer_32k"], seq_len=1024, budget=160, batch=2,
                  n_kv_heads=3, n_layers=2, group=group)
    A = 6
    (Ks, Vs, Qs), (Kd, Vd, Qdv) = make_inputs(w, sharpen_head=1)
    cfg = lib_config(w, budget_mode=R.RESKV_BUDGET_ADAKV, append_capacity=A)
    cache = R.reskv_build_cache(cfg, Kd, Vd, Qdv)
    budgets = R.reskv_get_unit_budgets(cache)
    assert budgets.reshape(-1, w.n_kv_heads).sum(axis=1).tolist() == [3 * 160] * (2 * 2)
    lay = R.reskv_export_cache(cache)
    assert np.array_equal(np.diff(lay["offsets"]), budgets + A)
    units = {u: unit_from_layout(lay, u) for u in range(w.n_units)}
    ocfg = lambda u: oracle_config(w, cfg, budgets[u], u)
    g = torch.Generator().manual_seed(5)
    for rnd in range(3):
        kn = torch.randn((w.n_layers, w.batch, w.n_kv_heads, 128), generator=g).to(torch.bfloat16)
        vn = torch.randn((w.n_layers, w.batch, w.n_kv_heads, 128), generator=g).to(torch.bfloat16)
        if rnd == 1:
            for l in range(w.n_layers):
                R.reskv_append(cache, l, kn[l].cuda().contiguous(), vn[l].cuda().contiguous())
        else:
            R.reskv_append(cache, -1, kn.cuda().contiguous(), vn.cuda().contiguous())
        kf, vf = bf16_to_f64(kn), bf16_to_f64(vn)
        for u in range(w.n_units):
            l, rem = divmod(u, w.batch * w.n_kv_heads)
            b, h = divmod(rem, w.n_kv_heads)
            units[u] = orc.append_tokens(units[u], kf[l, b, h][None], vf[l, b, h][None],
                                         np.array([w.seq_len + rnd]))
        # queries aimed at the newest token of every unit
        Q = torch.empty((w.n_layers, w.batch, w.n_q_heads, 128), dtype=torch.bfloat16)
        for l in range(w.n_layers):
            for b in range(w.batch):
                for h in range(w.n_kv_heads):
                    Q[l, b, h * group:(h + 1) * group] = (kn[l, b, h].float() * 0.5).to(torch.bfloat16)
        out = decode_all(cache, Q.cuda())
        lay2 = R.reskv_export_cache(cache)
        assert np.all(lay2["n_app"] == rnd + 1)
        compare_decode(out, Q, units, lay2, w, ocfg)
        O_l = np.zeros_like(out)
        for l in range(w.n_layers):
            Ol = torch.empty(Q.shape[1:], dtype=torch.float32, device="cuda")
            R.reskv_decode_attn(cache, l, Q[l].cuda().contiguous(), Ol)
            torch.cuda.synchronize()
            O_l[l] = Ol.cpu().numpy()
        compare_decode(O_l, Q, units, lay2, w, ocfg)
    cache.free()
