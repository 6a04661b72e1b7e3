"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test names the passage it follows.  None of them re-derives the oracle's
own formula: they use closed forms (App. A.1, A.2), fixed points the paper
states (Sec. 5.4: R empty gives eviction; Sec. 4.2: adding the exact residual
recovers full attention; Sec. 5.3: c_j = 1 gives an exact token), textbook
softmax through scipy (which the oracle does not call), explicit scalar loops
and hand-computed fixtures under ``tests/golden``.
"""
import json
import math
import os

import numpy as np
import pytest
from scipy.special import softmax

import oracle as orc
from paper_2607_29591_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def bf16ish(rng, shape, scale=1.0):
    """Random values that are exact bf16 numbers (8 significant bits)."""
    return orc.round_to_bf16(rng.standard_normal(shape) * scale)


def textbook_attention(q, K, V):
    """softmax(q K^T / sqrt(d)) V through scipy (Eq. attn / Eq. evict)."""
    w = softmax(K @ q / math.sqrt(K.shape[1]))
    return w @ V


# ---------------------------------------------------------------------------
# storage helpers
# ---------------------------------------------------------------------------

def test_bf16_rounding_fixture():
    g = golden("bf16_rounding.json")
    for c in g["cases"]:
        assert orc.round_to_bf16(np.array([c["x"]]))[0] == c["rounded"], c["note"]
    for c in g["bits"]:
        assert orc.bf16_bits_to_f64(np.array([c["bits"]], dtype=np.uint16))[0] == c["value"]


def test_bf16_rounding_is_idempotent_on_bf16_values():
    bits = np.arange(0, 1 << 16, 7, dtype=np.uint16)
    bits = bits[((bits >> 7) & 0xFF) != 0xFF]          # drop inf / NaN patterns
    vals = orc.bf16_bits_to_f64(bits)
    vals = vals[np.isfinite(vals) & (np.abs(vals) > 1e-30) & (np.abs(vals) < 1e30)]
    assert np.array_equal(orc.round_to_bf16(vals), vals)


# ---------------------------------------------------------------------------
# Decode (Alg. 2) fixed points and closed forms
# ---------------------------------------------------------------------------

def _cfg(**kw):
    base = dict(budget=8)
    base.update(kw)
    return orc.OracleConfig(**base)


def test_decode_empty_residual_is_eviction_attention():
    """Sec. 5.4: with R empty the shared softmax is eviction attention (Eq. evict)."""
    rng = np.random.default_rng(1)
    d, m = 16, 37
    K, V, q = bf16ish(rng, (m, d)), bf16ish(rng, (m, d)), bf16ish(rng, d, 2.0)
    out = orc.shared_softmax_decode(q, K, V, np.zeros((0, d)), np.zeros((0, d)),
                                    np.zeros(0), _cfg())
    np.testing.assert_allclose(out, textbook_attention(q, K, V), rtol=1e-12, atol=1e-13)


def test_decode_gate_zero_is_main_only():
    """Gate fixed to 0: log g = -inf removes every residual term (Eq. residual_logit)."""
    rng = np.random.default_rng(2)
    d, m, r = 16, 20, 6
    K, V, q = bf16ish(rng, (m, d)), bf16ish(rng, (m, d)), bf16ish(rng, d, 2.0)
    Kr, Vr = bf16ish(rng, (r, d)), bf16ish(rng, (r, d), 5.0)
    logc = np.log(rng.integers(1, 50, r).astype(float))
    out = orc.shared_softmax_decode(q, K, V, Kr, Vr, logc,
                                    _cfg(gate_mode=orc.GATE_FIXED, g_fixed=0.0))
    np.testing.assert_allclose(out, textbook_attention(q, K, V), rtol=1e-12, atol=1e-13)


def test_decode_exact_residual_encoding_recovers_full_attention():
    """Sec. 4.2, Eq. residual: adding (N_E, Z_E) back recovers o_S exactly.

    One residual entry whose logit carries log Z_E(q) and whose value is
    N_E/Z_E encodes the omitted statistics of q exactly; with g = 1 the shared
    softmax (Eqs. reskv_den, reskv_num) must equal full attention.  Z_E and N_E
    are summed here with explicit scalar loops.
    """
    rng = np.random.default_rng(3)
    d, s, m = 8, 40, 12
    K, V, q = bf16ish(rng, (s, d)), bf16ish(rng, (s, d)), bf16ish(rng, d, 1.5)
    M, E = np.arange(m), np.arange(m, s)
    ZE, NE = 0.0, np.zeros(d)
    for p in E:
        a = sum(q[i] * K[p, i] for i in range(d)) / math.sqrt(d)
        ZE += math.exp(a)
        NE += math.exp(a) * V[p]
    kbar = bf16ish(rng, (1, d))
    a_bar = float(kbar[0] @ q) / math.sqrt(d)
    logc = np.array([math.log(ZE) - a_bar])
    out = orc.shared_softmax_decode(q, K[M], V[M], kbar, (NE / ZE)[None, :], logc,
                                    _cfg(gate_mode=orc.GATE_FIXED, g_fixed=1.0))
    np.testing.assert_allclose(out, textbook_attention(q, K, V), rtol=1e-11, atol=1e-12)


def test_decode_weights_sum_to_one():
    """o^ = N^/Z^ is a convex combination: constant values come back unchanged."""
    rng = np.random.default_rng(4)
    d, m, r = 8, 10, 5
    c = bf16ish(rng, d)
    K, q = bf16ish(rng, (m, d)), bf16ish(rng, d)
    Kr = bf16ish(rng, (r, d))
    logc = np.log(np.arange(1, r + 1, dtype=float) * 3)
    out = orc.shared_softmax_decode(q, K, np.tile(c, (m, 1)), Kr, np.tile(c, (r, 1)), logc, _cfg())
    np.testing.assert_allclose(out, c, rtol=1e-13, atol=1e-14)


def test_decode_residual_mass_enters_both_numerator_and_denominator():
    """Eqs. reskv_den/reskv_num on a hand-sized case: one main token, one entry.

    Main: a_1 = 0, v = 0.  Entry: <q,k_bar>/sqrt(d) = 0, c = 3, g = 1, v_bar = 1:
    o^ = 3 * 1 / (1 + 3) = 0.75.
    """
    d = 4
    q = np.zeros(d)
    out = orc.shared_softmax_decode(q, np.zeros((1, d)), np.zeros((1, d)), np.zeros((1, d)),
                                    np.ones((1, d)), np.log([3.0]),
                                    _cfg(gate_mode=orc.GATE_FIXED, g_fixed=1.0))
    np.testing.assert_allclose(out, 0.75, rtol=1e-15)
    # the dynamic gate with a single main token: p_max = 1 -> g = sigmoid(-9)
    out2, st = orc.shared_softmax_decode(q, np.zeros((1, d)), np.zeros((1, d)), np.zeros((1, d)),
                                         np.ones((1, d)), np.log([3.0]), _cfg(), return_stats=True)
    g = 1.0 / (1.0 + math.exp(9.0))
    assert st["p_max"] == 1.0
    np.testing.assert_allclose(st["g"], g, rtol=1e-15)
    np.testing.assert_allclose(out2, 3 * g / (1 + 3 * g), rtol=1e-14)


def test_separate_softmax_hand_sized():
    """"w/o shared softmax" ablation (Table ablation_main), reading o^ = (1-g) o_M + g o_R.

    Main: one token with v = 0; one entry with v_bar = 1 and c = 3.  Each branch
    is normalised on its own, so o_R = 1 whatever c is, and o^ = g."""
    d = 4
    q = np.zeros(d)
    args = (q, np.zeros((1, d)), np.zeros((1, d)), np.zeros((1, d)), np.ones((1, d)), np.log([3.0]))
    for gf in (0.0, 0.3, 1.0):
        out = orc.separate_softmax_decode(*args, _cfg(gate_mode=orc.GATE_FIXED, g_fixed=gf,
                                                      softmax_mode=orc.SOFTMAX_SEPARATE))
        np.testing.assert_allclose(out, gf, rtol=1e-15, atol=0)
    out = orc.separate_softmax_decode(*args, _cfg(softmax_mode=orc.SOFTMAX_SEPARATE))
    np.testing.assert_allclose(out, 1.0 / (1.0 + math.exp(9.0)), rtol=1e-14)   # p_max = 1


def test_separate_softmax_single_entry_and_count_weighting():
    """Separate normalisations on random data: a single entry gives o_R = v_bar,
    so o^ = (1-g) o_M + g v_bar with the gate of the main logits; two entries
    with one key weigh their values by their counts (log c_j in the logit)."""
    rng = np.random.default_rng(21)
    d, m = 16, 30
    K, V, q = bf16ish(rng, (m, d)), bf16ish(rng, (m, d)), bf16ish(rng, d, 2.0)
    cfg = _cfg(softmax_mode=orc.SOFTMAX_SEPARATE)
    # gate by hand: p_max = largest main softmax weight
    a = [sum(q[i] * K[p, i] for i in range(d)) / math.sqrt(d) for p in range(m)]
    p_max = 1.0 / sum(math.exp(x - max(a)) for x in a)
    g = max(0.0, 1.0 / (1.0 + math.exp(-12.0 * (0.25 - p_max))))
    kb, vb = bf16ish(rng, (1, d)), bf16ish(rng, (1, d), 3.0)
    out = orc.separate_softmax_decode(q, K, V, kb, vb, np.log([7.0]), cfg)
    np.testing.assert_allclose(out, (1 - g) * textbook_attention(q, K, V) + g * vb[0],
                               rtol=1e-12, atol=1e-13)
    kb2 = np.vstack([kb, kb])
    vb2 = bf16ish(rng, (2, d), 3.0)
    out2 = orc.separate_softmax_decode(q, K, V, kb2, vb2, np.log([2.0, 6.0]), cfg)
    o_r = (2.0 * vb2[0] + 6.0 * vb2[1]) / 8.0
    np.testing.assert_allclose(out2, (1 - g) * textbook_attention(q, K, V) + g * o_r,
                               rtol=1e-12, atol=1e-13)
    # no residual mass (every c = 0): main-only, whatever g
    out3 = orc.separate_softmax_decode(q, K, V, kb2, vb2, np.array([-np.inf, -np.inf]), cfg)
    np.testing.assert_allclose(out3, textbook_attention(q, K, V), rtol=1e-12, atol=1e-13)
    # the dispatcher routes by softmax_mode
    np.testing.assert_allclose(orc.decode_query(q, K, V, kb, vb, np.log([7.0]), cfg), out, rtol=0)


def test_append_without_residual_is_attention_over_main_and_new_tokens():
    """Sec. 3.1 decode growth: tokens appended to a residual-free cache are
    attended exactly, so decode is textbook softmax attention over M plus the
    new tokens (Eq. attn on the grown cache)."""
    rng = np.random.default_rng(31)
    d, m, n = 16, 25, 3
    K, V = bf16ish(rng, (m + n, d)), bf16ish(rng, (m + n, d))
    q = bf16ish(rng, d, 2.0)
    base = orc.UnitCache(main_pos=np.arange(m), kmain=K[:m], vmain=V[:m], kbar=np.zeros((0, d)),
                         vbar=np.zeros((0, d)), counts=np.zeros(0, int), logc=np.zeros(0), r=0)
    grown = orc.append_tokens(base, K[m:], V[m:], np.arange(100, 100 + n))
    assert grown.main_pos.tolist() == list(range(m)) + [100, 101, 102]
    out = orc.decode_unit(grown, q[None, :], _cfg())[0]
    np.testing.assert_allclose(out, textbook_attention(q, K, V), rtol=1e-12, atol=1e-13)


def test_append_counts_in_the_gate_and_keeps_residual_entries():
    """An appended token with a dominant logit takes all main mass: p_max -> 1,
    so the dynamic gate falls to sigmoid(alpha (tau - 1)) (Eq. gate) and the
    residual entries, unchanged by the append, weigh in with that gate."""
    d = 4
    q = np.zeros(d)
    q[0] = 40.0
    Km = np.zeros((3, d))                        # three main tokens with logit 0
    Vm = np.zeros((3, d))
    kb, vb = np.zeros((1, d)), np.ones((1, d))   # one entry, logit log 5
    base = orc.UnitCache(main_pos=np.arange(3), kmain=Km, vmain=Vm, kbar=kb, vbar=vb,
                         counts=np.array([5]), logc=np.log([5.0]), r=1)
    k_new = np.zeros((1, d))
    k_new[0, 0] = 1.0                            # <q, k_new>/sqrt(d) = 20
    v_new = np.full((1, d), 2.0)
    grown = orc.append_tokens(base, k_new, v_new, np.array([7]))
    assert grown.r == 1 and np.array_equal(grown.kbar, kb) and grown.logc[0] == math.log(5.0)
    out, st = orc.shared_softmax_decode(q, grown.kmain, grown.vmain, grown.kbar, grown.vbar,
                                        grown.logc, _cfg(), return_stats=True)
    e20 = math.exp(20.0)
    p_max = e20 / (3.0 + e20)
    g = 1.0 / (1.0 + math.exp(-12.0 * (0.25 - p_max)))
    np.testing.assert_allclose(st["p_max"], p_max, rtol=1e-15)
    np.testing.assert_allclose(st["g"], g, rtol=1e-12)
    expect = (e20 * 2.0 + 5.0 * g * 1.0) / (3.0 + e20 + 5.0 * g)
    np.testing.assert_allclose(out, expect, rtol=1e-14)


def test_gate_closed_forms():
    """Eq. gate with the paper's tau = 0.25, alpha = 12 (App. B), via uniform main caches."""
    gc = golden("gate_closed_forms.json")
    for c in gc["cases"]:
        assert orc.dynamic_gate(c["p_max"], 0.25, 12.0, 0.0) == pytest.approx(c["g"], rel=1e-14)
    cm = gc["g_min_case"]
    assert orc.dynamic_gate(cm["p_max"], 0.25, 12.0, cm["g_min"]) == cm["g"]
    # through the decode path: m identical keys give p_max = 1/m
    d = 4
    q = np.ones(d)
    for m, case in ((4, 0), (1, 1), (8, 2), (2, 3)):
        K = np.tile(np.array([0.5, -1.0, 0.25, 2.0]), (m, 1))
        _, st = orc.shared_softmax_decode(q, K, np.zeros((m, d)), np.zeros((1, d)), np.zeros((1, d)),
                                          np.zeros(1), _cfg(), return_stats=True)
        assert st["p_max"] == pytest.approx(1.0 / m, rel=1e-15)
        assert st["g"] == pytest.approx(gc["cases"][case]["g"], rel=1e-13)


def test_eviction_error_closed_form():
    """App. A.1, Eq. app_evict_error: o_S - o_M = (Z_M N_E - Z_E N_M) / (Z_M (Z_M + Z_E))."""
    rng = np.random.default_rng(5)
    d, s, m = 8, 50, 15
    K, V, q = bf16ish(rng, (s, d)), bf16ish(rng, (s, d)), bf16ish(rng, d, 1.5)
    M, E = np.arange(m), np.arange(m, s)
    ZM = sum(math.exp(float(K[p] @ q) / math.sqrt(d)) for p in M)
    NM = sum(math.exp(float(K[p] @ q) / math.sqrt(d)) * V[p] for p in M)
    ZE = sum(math.exp(float(K[p] @ q) / math.sqrt(d)) for p in E)
    NE = sum(math.exp(float(K[p] @ q) / math.sqrt(d)) * V[p] for p in E)
    closed = (ZM * NE - ZE * NM) / (ZM * (ZM + ZE))
    o_S = orc.attention_full(q, K, V)
    o_M = orc.shared_softmax_decode(q, K[M], V[M], np.zeros((0, d)), np.zeros((0, d)),
                                    np.zeros(0), _cfg())
    np.testing.assert_allclose(o_S - o_M, closed, rtol=1e-10, atol=1e-13)


def test_entry_error_bound():
    """App. A.2: |Z_j - c_j e^{a_bar}| <= c_j e^{a_bar} (e^eta - 1) and the
    numerator bound with V = max ||v_p||, for the entry the oracle builds."""
    rng = np.random.default_rng(6)
    d, c = 16, 30
    centre = bf16ish(rng, d)
    for spread in (0.01, 0.1, 0.5):
        KC = centre + spread * rng.standard_normal((c, d))
        VC = rng.standard_normal((c, d))
        q = rng.standard_normal(d)
        E = np.arange(c)
        kbar, vbar, counts = orc.lloyd_residual(KC, VC, E, 1, 4)
        assert counts[0] == c
        # the entry's reconstructed statistics, read from the shared softmax
        main_k = np.zeros((1, d))
        _, st = orc.shared_softmax_decode(q, main_k, np.zeros((1, d)), kbar, vbar,
                                          orc.log_counts(counts, 1.0),
                                          _cfg(gate_mode=orc.GATE_FIXED, g_fixed=1.0),
                                          return_stats=True)
        Z_hat = st["Z"] * math.exp(st["shift"]) - 1.0          # minus the main token's e^0
        N_hat = st["N"] * math.exp(st["shift"])                 # main value is 0
        a = KC @ q / math.sqrt(d)
        a_bar = float(kbar[0] @ q) / math.sqrt(d)
        eta = float(np.max(np.abs(a - a_bar)))
        Zj = float(np.sum(np.exp(a)))
        Nj = np.exp(a) @ VC
        bound_z = c * math.exp(a_bar) * (math.exp(eta) - 1)
        Vmax = float(np.max(np.linalg.norm(VC, axis=1)))
        np.testing.assert_allclose(Z_hat, c * math.exp(a_bar), rtol=1e-12)
        assert abs(Zj - Z_hat) <= bound_z * (1 + 1e-12)
        assert np.linalg.norm(Nj - N_hat) <= bound_z * Vmax * (1 + 1e-12)


# ---------------------------------------------------------------------------
# Selection (Sec. 5.2) and candidate budgets (App. B)
# ---------------------------------------------------------------------------

def test_ranking_and_selection_fixture():
    g = golden("ranking_ties.json")
    ranked = orc.rank_evictable(np.array(g["scores"]), g["recent"])
    assert ranked.tolist() == g["ranked"]
    M, E = orc.select_main(ranked, len(g["scores"]), g["recent"], g["m"])
    assert M.tolist() == g["M"]
    assert E.tolist() == g["E_rank_order"]


def test_ranking_matches_brute_force_order():
    """Brute force: a scalar insertion sort by (score desc, index asc)."""
    rng = np.random.default_rng(7)
    for trial in range(20):
        s = int(rng.integers(1, 30))
        recent = int(rng.integers(0, 6))
        scores = rng.integers(0, 5, s).astype(float)     # many exact ties
        ranked = orc.rank_evictable(scores, recent)
        out = []
        for p in range(max(s - recent, 0)):
            i = 0
            while i < len(out) and (scores[out[i]] > scores[p] or
                                    (scores[out[i]] == scores[p] and out[i] < p)):
                i += 1
            out.insert(i, p)
        assert ranked.tolist() == out


def test_candidate_budgets_fixture():
    g = golden("candidate_budgets.json")
    for b, rs in g["cases"].items():
        assert orc.candidate_budgets(int(b), g["ratios"]) == rs


def test_choose_r_rules():
    """Eq. valproxy: argmin over r > 0 (ties -> smaller r), strict margin test."""
    rs = [25, 51, 76, 102]
    assert orc.choose_r(1.0, rs, [0.5, 0.4, 0.4, 0.6], 0.01) == 51
    assert orc.choose_r(1.0, rs, [0.995] * 4, 0.01) == 0
    assert orc.choose_r(1.0, rs, [0.99, 1.0, 1.1, 1.2], 0.01) == 0   # equality is not enough
    assert orc.choose_r(1.0, rs, [0.98, 1.0, 1.1, 1.2], 0.01) == 25
    assert orc.choose_r(0.0, rs, [0.0] * 4, 0.01) == 0
    assert orc.choose_r(1.0, [], [], 0.01) == 0


# ---------------------------------------------------------------------------
# Residual construction (Sec. 5.3)
# ---------------------------------------------------------------------------

def test_lloyd_hand_traces():
    g = golden("lloyd_traces.json")
    for c in g["cases"]:
        K = np.array(c["keys"], dtype=float)[:, None]
        V = 2 * K + 1
        kbar, vbar, counts = orc.lloyd_residual(K, V, np.array(c["E"]), c["r"], c["iters"])
        np.testing.assert_allclose(kbar[:, 0], c["kbar"], rtol=1e-15, err_msg=c["name"])
        assert counts.tolist() == c["counts"], c["name"]
        for j in range(c["r"]):
            if counts[j] > 0:
                assert vbar[j, 0] == pytest.approx(2 * kbar[j, 0] + 1, rel=1e-14), c["name"]
            else:
                assert vbar[j, 0] == 0.0


def test_lloyd_single_entry_is_global_mean():
    rng = np.random.default_rng(8)
    K, V = rng.standard_normal((57, 6)), rng.standard_normal((57, 6))
    E = rng.permutation(57)[:40]
    kbar, vbar, counts = orc.lloyd_residual(K, V, E, 1, 4)
    np.testing.assert_allclose(kbar[0], K[E].mean(axis=0), rtol=1e-13)
    np.testing.assert_allclose(vbar[0], V[E].mean(axis=0), rtol=1e-13)
    assert counts.tolist() == [40]


def test_lloyd_separated_clusters_converge_to_true_means():
    rng = np.random.default_rng(9)
    d, per = 8, 25
    centres = 50.0 * np.eye(d)[:3]
    K = np.concatenate([c + rng.standard_normal((per, d)) for c in centres])
    V = rng.standard_normal((3 * per, d))
    E = np.array([0, per, 2 * per] + [p for p in range(3 * per) if p % per])
    kbar, vbar, counts = orc.lloyd_residual(K, V, E, 3, 4)
    for j in range(3):
        np.testing.assert_allclose(kbar[j], K[j * per:(j + 1) * per].mean(axis=0), rtol=1e-12)
        np.testing.assert_allclose(vbar[j], V[j * per:(j + 1) * per].mean(axis=0), rtol=1e-12)
    assert counts.tolist() == [per] * 3


def test_lloyd_assign_matches_direct_distances():
    """The matrix-product form of the distance picks the same centre as a
    direct sum of squared differences (scalar loops)."""
    rng = np.random.default_rng(10)
    KE = bf16ish(rng, (60, 5))
    C = bf16ish(rng, (7, 5))
    got = orc.lloyd_assign(KE, C)
    for p in range(KE.shape[0]):
        best, bd = 0, None
        for j in range(C.shape[0]):
            dd = sum((KE[p, i] - C[j, i]) ** 2 for i in range(5))
            if bd is None or dd < bd:
                best, bd = j, dd
        assert got[p] == best


def test_exact_groups_reproduce_full_attention():
    """Sec. 5.3 / App. A.2 with eta = 0: an entry with c_j = 1 is an exact token,
    and a group of c_j identical tokens is reconstructed exactly (c_j e^{a_bar}
    equals the group's sum).  With every evicted group exact and g = 1 the
    shared softmax is full attention over S."""
    rng = np.random.default_rng(11)
    d, m = 16, 20
    # singletons: r = |E|, every key distinct
    K, V = bf16ish(rng, (m + 12, d)), bf16ish(rng, (m + 12, d))
    E = np.arange(m, m + 12)[::-1]
    kbar, vbar, counts = orc.lloyd_residual(K, V, E, len(E), 4)
    assert counts.tolist() == [1] * len(E)
    np.testing.assert_array_equal(kbar, K[E])
    cfg = orc.OracleConfig(budget=m + 12, gate_mode=orc.GATE_FIXED, g_fixed=1.0)
    for _ in range(4):
        q = bf16ish(rng, d, 1.5)
        out = orc.shared_softmax_decode(q, K[:m], V[:m], kbar, vbar, orc.log_counts(counts, 1.0), cfg)
        np.testing.assert_allclose(out, textbook_attention(q, K, V), rtol=1e-11, atol=1e-12)
    # groups of identical tokens: 5 prototypes repeated 1..5 times
    protos_k, protos_v = bf16ish(rng, (5, d)), bf16ish(rng, (5, d))
    reps = [3, 1, 5, 2, 4]
    KE = np.concatenate([np.tile(protos_k[i], (reps[i], 1)) for i in range(5)])
    VE = np.concatenate([np.tile(protos_v[i], (reps[i], 1)) for i in range(5)])
    K2 = np.concatenate([K[:m], KE])
    V2 = np.concatenate([V[:m], VE])
    firsts = np.cumsum([0] + reps[:-1]) + m
    rest = [p for p in range(m, m + sum(reps)) if p not in set(firsts.tolist())]
    E2 = np.concatenate([firsts, rest])                 # one of each prototype first
    kbar, vbar, counts = orc.lloyd_residual(K2, V2, E2, 5, 4)
    assert counts.tolist() == reps
    for _ in range(4):
        q = bf16ish(rng, d, 1.5)
        out = orc.shared_softmax_decode(q, K2[:m], V2[:m], kbar, vbar,
                                        orc.log_counts(counts, 1.0), cfg)
        np.testing.assert_allclose(out, textbook_attention(q, K2, V2), rtol=1e-11, atol=1e-12)


# ---------------------------------------------------------------------------
# Scoring (App. B.2)
# ---------------------------------------------------------------------------

def test_scores_uniform_keys():
    """Identical keys give uniform weights 1/s per query and head; the sum over
    n_fit queries is n_fit/s, and the zero-padded pool of width 5 keeps 3/5 and
    4/5 of it at the two ends."""
    s, d, G, n_fit = 20, 4, 3, 7
    K = np.tile(np.array([0.5, 1.0, -2.0, 0.25]), (s, 1))
    Q = np.random.default_rng(12).standard_normal((G, n_fit, d))
    sc = orc.scores_obs_pool(K, Q, 5)
    base = n_fit / s
    expect = np.full(s, base)
    expect[[0, -1]] = base * 3 / 5
    expect[[1, -2]] = base * 4 / 5
    np.testing.assert_allclose(sc, expect, rtol=1e-13)


def test_scores_single_peak_pooling_and_head_average():
    """One key with logit L (others 0) per head: weight e^L/(e^L + s - 1) at
    that token.  Two heads peaked at different tokens average with 1/G, fit
    queries sum, and the pool spreads each peak over 5 neighbours.  The
    validation rows (not passed) play no part."""
    s, d = 30, 2
    K = np.zeros((s, d))
    K[10, 0] = 4.0
    K[20, 1] = 6.0
    n_fit = 3
    Q = np.zeros((2, n_fit, d))
    Q[0, :, 0] = 2.0
    Q[1, :, 1] = 1.0
    L0, L1 = 4.0 * 2.0 / math.sqrt(2), 6.0 * 1.0 / math.sqrt(2)
    w0 = math.exp(L0) / (math.exp(L0) + s - 1)
    w1 = math.exp(L1) / (math.exp(L1) + s - 1)
    A = np.zeros(s)
    A += n_fit * 0.5 * np.where(np.arange(s) == 10, w0, (1 - w0) / (s - 1))
    A += n_fit * 0.5 * np.where(np.arange(s) == 20, w1, (1 - w1) / (s - 1))
    expect = np.array([sum(A[p + j] for j in range(-2, 3) if 0 <= p + j < s) / 5 for p in range(s)])
    np.testing.assert_allclose(orc.scores_obs_pool(K, Q, 5), expect, rtol=1e-12)


def test_build_uses_only_fit_rows_for_scores():
    rng = np.random.default_rng(13)
    s, d = 64, 8
    K, V = bf16ish(rng, (s, d)), bf16ish(rng, (s, d))
    Q = bf16ish(rng, (2, 10, d))
    cfg = orc.OracleConfig(budget=24, recent_window=4, n_fit=7, n_val=3, residual_override=4)
    a = orc.build_unit(K, V, Q, cfg)
    Q2 = Q.copy()
    Q2[:, 7:] = bf16ish(rng, (2, 3, d), 3.0)
    b = orc.build_unit(K, V, Q2, cfg)
    np.testing.assert_array_equal(a.scores, b.scores)
    np.testing.assert_array_equal(a.main_pos, b.main_pos)


def test_keynorm_scores():
    K = np.array([[1.0, 2.0], [3.0, -1.0], [0.0, 0.5]])
    np.testing.assert_array_equal(orc.scores_keynorm(K), [5.0, 10.0, 0.25])


def test_keynorm_score_is_the_exact_sum_rounded_once():
    """A row of bf16 values whose squares span more than 53 bits: 2^14 in the
    first dim (square 2^28, ulp 2^-24) and 2^-13 in the other 127 (squares
    2^-26, a quarter ulp each).  Summed in dim order, every small square is
    rounded away and the sum stays 2^28; the exact sum 2^28 + 127 * 2^-26
    rounds to 2^28 + 32 * 2^-24 = 2^28 + 2^-19.  The score must be the
    latter in every dim order."""
    row = np.full(128, 2.0 ** -13)
    row[0] = 2.0 ** 14
    in_order = 0.0
    for x in row:
        in_order += x * x
    assert in_order == 2.0 ** 28                      # what in-order summation gives
    want = 2.0 ** 28 + 2.0 ** -19
    K = np.stack([row, row[::-1], np.roll(row, 37)])
    np.testing.assert_array_equal(orc.scores_keynorm(K), [want, want, want])
    # exact integer arithmetic on the same squares agrees (every square of a
    # bf16 value is a dyadic rational: scale by 2^26 to integers)
    exact = sum(int(x * x * 2.0 ** 26) for x in row)
    assert exact == 2 ** 54 + 127 and float(exact) * 2.0 ** -26 == want


def test_keynorm_score_independent_of_dim_order_on_generator_rows():
    """On rows drawn like the workloads' keys (with outlier channels), any
    permutation of the dims gives the same score bit for bit, and the score
    equals the exact rational sum rounded once."""
    from fractions import Fraction
    w = wl.scaled(wl.WORKLOADS["small_budget_b64"], seq_len=64)
    K, _ = wl.unit_kv(w, 3, 1, 5)
    Kf = K.double().numpy()
    base = orc.scores_keynorm(Kf)
    rng = np.random.default_rng(8)
    for _ in range(3):
        np.testing.assert_array_equal(orc.scores_keynorm(Kf[:, rng.permutation(128)]), base)
    for p in range(0, 64, 9):
        exact = sum(Fraction(float(x)) ** 2 for x in Kf[p])
        assert float(exact) == base[p]


# ---------------------------------------------------------------------------
# Construction (Alg. 1) and the validation proxy (Sec. 5.5.1)
# ---------------------------------------------------------------------------

def test_budget_covering_every_token_is_full_attention():
    """b >= s: M = S, E empty, r = 0, and decode is full attention (Eq. attn)."""
    rng = np.random.default_rng(14)
    s, d = 30, 8
    K, V = bf16ish(rng, (s, d)), bf16ish(rng, (s, d))
    Q = bf16ish(rng, (4, 12, d))
    cfg = orc.OracleConfig(budget=32, recent_window=4, n_fit=8, n_val=4)
    cache = orc.build_unit(K, V, Q, cfg)
    assert cache.r == 0 and cache.main_pos.tolist() == list(range(s))
    q = bf16ish(rng, d)
    np.testing.assert_allclose(orc.decode_unit(cache, q[None], cfg)[0],
                               textbook_attention(q, K, V), rtol=1e-12, atol=1e-13)


def test_validation_loss_r0_matches_eviction_closed_form():
    """L_0 (Eq. valloss on the pure-main cache) equals the mean of ||o_S - o_M||^2
    written with the App. A.1 closed form."""
    rng = np.random.default_rng(15)
    s, d, G = 80, 8, 2
    K, V = bf16ish(rng, (s, d)), bf16ish(rng, (s, d))
    Q = bf16ish(rng, (G, 10, d), 1.5)
    cfg = orc.OracleConfig(budget=20, recent_window=4, n_fit=6, n_val=4)
    cache = orc.build_unit(K, V, Q, cfg)
    c0 = orc.build_candidate(K, V, cache.ranked, cfg, 0)
    M = c0.main_pos
    E = np.setdiff1d(np.arange(s), M)
    tot = 0.0
    for g in range(G):
        for t in range(6, 10):
            q = Q[g, t]
            e = np.exp(K @ q / math.sqrt(d))
            ZM, ZE = e[M].sum(), e[E].sum()
            NM, NE = e[M] @ V[M], e[E] @ V[E]
            diff = (ZM * NE - ZE * NM) / (ZM * (ZM + ZE))
            tot += float(diff @ diff)
    assert cache.losses[0] == pytest.approx(tot / (G * 4), rel=1e-10)


def test_validation_proxy_enables_residual_on_clusterable_diffuse_attention():
    """Evicted keys that form a few tight clusters under diffuse attention are
    reconstructed well, so L_r* beats L_0 by more than delta and r* > 0."""
    rng = np.random.default_rng(16)
    d, s = 8, 400
    protos = bf16ish(rng, (4, d), 0.6)
    K = np.concatenate([protos[i % 4] + 0.0 for i in range(s)]).reshape(s, d)
    V = np.concatenate([np.full(d, float(i % 4)) for i in range(s)]).reshape(s, d)
    K[: s // 2] = bf16ish(rng, (s // 2, d), 0.6)      # unclustered half, scored high
    Q = bf16ish(rng, (2, 16, d), 0.3)
    cfg = orc.OracleConfig(budget=100, recent_window=8, n_fit=12, n_val=4)
    cache = orc.build_unit(K, V, Q, cfg)
    assert cache.r > 0
    assert cache.losses[cache.r] < (1 - cfg.delta) * cache.losses[0]


def test_validation_proxy_falls_back_when_nothing_is_evicted():
    rng = np.random.default_rng(17)
    s, d = 24, 4
    K, V = bf16ish(rng, (s, d)), bf16ish(rng, (s, d))
    Q = bf16ish(rng, (1, 8, d))
    cache = orc.build_unit(K, V, Q, orc.OracleConfig(budget=24, recent_window=4, n_fit=6, n_val=2))
    assert cache.r == 0 and len(cache.main_pos) == s


# ---------------------------------------------------------------------------
# AdaKV budgets across KV heads (App. B, "AdaKV"; "+ResKV" rows of
# Table ruler_paper and Table longbench_paper)
# ---------------------------------------------------------------------------

def test_adakv_budgets_fixture():
    g = golden("adakv_budgets.json")
    for case in g["cases"]:
        got = orc.adakv_budgets(np.array(case["scores"]), g["budget"], g["recent"],
                                case["safeguard"])
        assert got.tolist() == case["budgets"], case["note"]


def _best_allocation(scores, budget, recent, f):
    """Exhaustive search: the split x_h >= f, sum x_h = H*(b - |P|), that keeps
    the largest total score (each head keeps its top x_h evictable tokens)."""
    H, s = scores.shape
    n_p = min(recent, s)
    n = budget - n_p
    tops = [np.concatenate([[0.0], np.cumsum(np.sort(scores[h, :s - n_p])[::-1])])
            for h in range(H)]
    best, arg = -1.0, None

    def rec(h, left, acc, xs):
        nonlocal best, arg
        if h == H - 1:
            if f <= left <= s - n_p:
                tot = acc + tops[h][left]
                if tot > best:
                    best, arg = tot, xs + [left]
            return
        for x in range(f, min(left, s - n_p) + 1):
            rec(h + 1, left - x, acc + tops[h][x], xs + [x])

    rec(0, H * n, 0.0, [])
    return np.array(arg) + n_p


@pytest.mark.parametrize("seed,H,s,recent,budget,safeguard",
                         [(0, 3, 12, 2, 5, 0.2), (1, 3, 12, 2, 5, 0.5), (2, 2, 16, 3, 7, 0.2),
                          (3, 4, 10, 1, 4, 0.34), (4, 3, 9, 0, 3, 0.0)])
def test_adakv_budgets_maximise_kept_score(seed, H, s, recent, budget, safeguard):
    """With distinct scores the allocation is the unique split (every head
    above its safeguard) that keeps the largest total score: each head's
    retained mass is concave in its budget, so the pooled pick of the best
    remaining tokens is optimal -- checked here by enumerating every split."""
    rng = np.random.default_rng(seed)
    scores = rng.random((H, s))
    n = budget - min(recent, s)
    f = int(np.floor(float(np.float32(safeguard)) * n))
    got = orc.adakv_budgets(scores, budget, recent, safeguard)
    assert got.tolist() == _best_allocation(scores, budget, recent, f).tolist()


def test_adakv_budgets_invariants_and_closed_forms():
    rng = np.random.default_rng(7)
    H, s, recent, b = 8, 300, 16, 64
    scores = rng.random((H, s))
    for sg in (0.0, 0.2, 0.5, 0.9):
        got = orc.adakv_budgets(scores, b, recent, sg)
        f = int(np.floor(float(np.float32(sg)) * (b - recent)))
        assert got.sum() == H * b and np.all(got >= recent + f) and np.all(got <= s)
    # safeguard 1: nothing is shared; identical heads: the pooled pick alternates
    assert orc.adakv_budgets(scores, b, recent, 1.0).tolist() == [b] * H
    assert orc.adakv_budgets(np.tile(scores[:1], (H, 1)), b, recent, 0.2).tolist() == [b] * H
    # the budget covers every token: no allocation
    assert orc.adakv_budgets(scores, s + 5, recent, 0.2).tolist() == [s + 5] * H
    # one dominant head takes every shared slot, b_3 = |P| + f + H (b - |P| - f),
    # as long as it has that many tokens; with fewer it keeps all s of them
    dom = rng.random((H, 500))
    dom[3] += 1000.0
    f = int(np.floor(float(np.float32(0.2)) * (b - recent)))
    got = orc.adakv_budgets(dom, b, recent, 0.2)
    assert got[3] == recent + f + H * (b - recent - f)
    assert all(got[h] == recent + f for h in range(H) if h != 3)
    got = orc.adakv_budgets(dom[:, :300], b, recent, 0.2)
    assert got[3] == 300 and got.sum() == H * b


def test_adakv_safeguard_one_is_uniform_resKV():
    """safeguard 1 leaves every head its uniform budget, so the grouped build is
    Alg. 1 per head unchanged."""
    rng = np.random.default_rng(3)
    H, s, d, G = 2, 96, 128, 2
    Ks = np.round(rng.standard_normal((H, s, d)) * 8) / 8
    Vs = np.round(rng.standard_normal((H, s, d)) * 8) / 8
    Qo = np.round(rng.standard_normal((H, G, 12, d)) * 8) / 8
    cfgs = [orc.OracleConfig(budget=32, recent_window=8, n_fit=8, n_val=4)] * H
    budgets, units = orc.build_heads_adakv(Ks, Vs, Qo, cfgs, 1.0)
    assert budgets.tolist() == [32, 32]
    for h in range(H):
        ref = orc.build_unit(Ks[h], Vs[h], Qo[h], cfgs[h])
        assert ref.r == units[h].r
        assert np.array_equal(ref.main_pos, units[h].main_pos)
        assert np.array_equal(ref.kbar, units[h].kbar)


def test_adakv_grouped_build_keeps_each_heads_budget():
    """Every head's cache fills exactly its allocated budget b_h = m_h + r_h,
    keeps its window, and its main tokens are its top b_h - |P| ranked tokens."""
    rng = np.random.default_rng(5)
    H, s, d, G = 3, 160, 128, 2
    Ks = np.round(rng.standard_normal((H, s, d)) * 8) / 8
    Ks[1] *= 3.0                      # a sharper head attracts budget
    Vs = np.round(rng.standard_normal((H, s, d)) * 8) / 8
    Qo = np.concatenate([Ks[:, None, rng.integers(0, s, 12)], Ks[:, None, rng.integers(0, s, 12)]],
                        axis=1) + 0.1
    cfgs = [orc.OracleConfig(budget=40, recent_window=8, n_fit=8, n_val=4)] * H
    budgets, units = orc.build_heads_adakv(Ks, Vs, Qo, cfgs, 0.2)
    assert budgets.sum() == H * 40
    for h in range(H):
        u = units[h]
        assert len(u.main_pos) + u.r == budgets[h]
        assert set(range(s - 8, s)) <= set(u.main_pos.tolist())
        keep = len(u.main_pos) - 8
        assert set(u.ranked[:keep].tolist()) | set(range(s - 8, s)) == set(u.main_pos.tolist())


# ---------------------------------------------------------------------------
# Decode-time growth into a bounded region (Sec. 3.1; App. E refresh)
# ---------------------------------------------------------------------------

def test_nearest_entry_is_exact_with_ties_to_the_lower_entry():
    d = 128
    k = np.zeros(d)
    # squared distances 2^54 + 1 and 2^54 + 1/4: equal once rounded to float64
    # (ulp 4 at 2^54), so only the exact comparison finds entry 1
    kbar = np.zeros((2, d))
    kbar[:, 0] = 2.0 ** 27
    kbar[0, 1], kbar[1, 1] = 1.0, 0.5
    fp64 = np.sum((kbar - k) ** 2, axis=1)
    assert fp64[0] == fp64[1]
    assert orc.nearest_entry(k, kbar) == 1
    # exact ties go to the lower entry; k midway between two entries
    kbar = np.zeros((3, d))
    kbar[0, 3], kbar[1, 3], kbar[2, 3] = 1.0, -1.0, 1.0
    assert orc.nearest_entry(k, kbar) == 0
    assert orc.nearest_entry(k, kbar[[1, 0, 2]]) == 0
    # brute force on separated random entries agrees with a float64 argmin
    rng = np.random.default_rng(21)
    for _ in range(20):
        kb = orc.round_to_bf16(rng.normal(size=(7, d)) * 3)
        kk = orc.round_to_bf16(kb[rng.integers(7)] + rng.normal(size=d) * 0.1)
        assert orc.nearest_entry(kk, kb) == int(np.argmin(np.sum((kb - kk) ** 2, axis=1)))
    # bf16 subnormals take part exactly
    kbar = np.zeros((2, d))
    kbar[0, 0], kbar[1, 0] = 3 * 2.0 ** -133, 2.0 ** -133
    assert orc.nearest_entry(np.zeros(d), kbar) == 1


def test_fold_is_the_running_mean_stored_in_bf16():
    d = 128
    z = np.zeros(d)
    k = np.full(d, 0.75)
    kb, vb, c, lc = orc.fold_into_entry(z, z, 0, k, -k, 1.0)      # empty entry: the token
    assert np.array_equal(kb, k) and np.array_equal(vb, -k) and c == 1 and lc == 0.0
    kb, vb, c, lc = orc.fold_into_entry(np.ones(d), np.full(d, 2.0), 3, np.full(d, 5.0),
                                        np.full(d, -6.0), 1.0)
    assert np.all(kb == 2.0) and np.all(vb == 0.0) and c == 4       # (3+5)/4, (6-6)/4
    assert lc == pytest.approx(np.log(4.0), rel=0, abs=0)
    # (2 * 1 + 2) / 3 = 4/3 = 1.0101010101...b: bf16 keeps 1.0101011b = 1.3359375
    kb, _, _, lc = orc.fold_into_entry(np.ones(d), z, 2, np.full(d, 2.0), z, 0.5)
    assert np.all(kb == 1.3359375) and lc == 0.5 * np.log(3.0)


def _small_unit(rng, m, r, d=16, s_tokens=None):
    K = bf16ish(rng, (m + r, d))
    V = bf16ish(rng, (m + r, d))
    counts = rng.integers(1, 9, r)
    return orc.UnitCache(main_pos=np.arange(m), kmain=K[:m], vmain=V[:m], kbar=K[m:],
                         vbar=V[m:], counts=counts, logc=np.log(counts.astype(np.float64)), r=r)


def test_ring_append_keeps_the_most_recent_tokens():
    rng = np.random.default_rng(22)
    base = _small_unit(rng, 10, 0)
    A, n = 3, 8
    Kn, Vn = bf16ish(rng, (n, 16)), bf16ish(rng, (n, 16))
    pos = np.arange(100, 100 + n)
    # with room the ring is plain growth
    grown, na = orc.append_ring(base, Kn[:A], Vn[:A], pos[:A], 0, A, orc.APPEND_RING_DROP)
    ref = orc.append_tokens(base, Kn[:A], Vn[:A], pos[:A])
    assert na == A and np.array_equal(grown.kmain, ref.kmain)
    for policy in (orc.APPEND_RING_DROP, orc.APPEND_RING_FOLD):   # no entries: both drop
        out, na = orc.append_ring(base, Kn, Vn, pos, 0, A, policy)
        assert na == A
        assert np.array_equal(out.main_pos, np.concatenate([np.arange(10), pos[-A:]]))
        assert np.array_equal(out.kmain[-A:], Kn[-A:]) and np.array_equal(out.vmain[-A:], Vn[-A:])
        q = bf16ish(rng, 16)
        np.testing.assert_allclose(orc.decode_unit(out, q[None], orc.OracleConfig(budget=1))[0],
                                   textbook_attention(q, out.kmain, out.vmain), rtol=1e-12)
    with pytest.raises(ValueError):
        orc.append_ring(base, Kn, Vn, pos, 0, A, orc.APPEND_FAIL)


def test_ring_fold_loses_no_token_and_updates_the_nearest_entry():
    rng = np.random.default_rng(23)
    m, r, A = 12, 4, 5
    base = _small_unit(rng, m, r)
    before = base.counts.sum() + m
    Kn, Vn = bf16ish(rng, (3 * A, 16)), bf16ish(rng, (3 * A, 16))
    out, na = orc.append_ring(base, Kn, Vn, np.arange(50, 50 + 3 * A), 0, A,
                              orc.APPEND_RING_FOLD)
    assert na == A and out.kmain.shape[0] == m + A
    assert out.counts.sum() + out.kmain.shape[0] == before + 3 * A       # every token kept
    # the first token to leave (appended first) went to its nearest entry
    one, _ = orc.append_ring(base, Kn[:A + 1], Vn[:A + 1], np.arange(A + 1), 0, A,
                             orc.APPEND_RING_FOLD)
    j = orc.nearest_entry(Kn[0], base.kbar)
    assert one.counts[j] == base.counts[j] + 1
    assert np.array_equal(np.delete(one.counts, j), np.delete(base.counts, j))
    want = orc.round_to_bf16((base.counts[j] * base.kbar[j] + Kn[0]) / (base.counts[j] + 1))
    assert np.array_equal(one.kbar[j], want)
    assert one.logc[j] == np.log(base.counts[j] + 1.0)


def test_bf16_rounding_in_the_subnormal_range():
    """Below 2^-126 bf16 values are multiples of 2^-133: 2^-134 is a tie
    between 0 and 2^-133 (to even: 0), 3 * 2^-134 a tie between 2^-133 and
    2 * 2^-133 (to even: 2^-132), 1.25 * 2^-133 rounds down to 2^-133; the
    smallest normal 2^-126 and its neighbours keep 8 significant bits."""
    t = 2.0 ** -133
    got = orc.round_to_bf16(np.array([2.0 ** -134, 3 * 2.0 ** -134, 1.25 * t, -1.75 * t,
                                      2.0 ** -126, 2.0 ** -126 * (1 + 2.0 ** -8),
                                      2.0 ** -126 * (1 + 3 * 2.0 ** -8), 127.5 * t]))
    want = [0.0, 2.0 ** -132, t, -2 * t, 2.0 ** -126, 2.0 ** -126,
            2.0 ** -126 * (1 + 2 * 2.0 ** -7), 128 * t]
    assert got.tolist() == want
    # every value the bf16 format holds is left alone
    bits = np.arange(0, 0x7f80, 7, dtype=np.uint16)
    vals = orc.bf16_bits_to_f64(bits)
    assert np.array_equal(orc.round_to_bf16(vals), vals)
