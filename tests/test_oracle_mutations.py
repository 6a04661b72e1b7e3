"""Plant plausible mistakes in the oracle (on the CPU) and check that the pins
of tests/test_oracle_pins.py catch every one of them.

Each mutant replaces one oracle function with a version carrying a single
mistake of the kind that slips into a restatement of the paper: a dropped
term, a wrong sign, scale or index, a tie broken the other way, a missing
normalisation.  A mutant survives if every pin still passes; none may.
"""
import contextlib
import inspect

import numpy as np
import pytest

import oracle
import oracle.reskv_oracle as core
import test_oracle_pins as pins


@contextlib.contextmanager
def patched(name, fn):
    """Replace `name` in the oracle module and in the package re-export."""
    old = getattr(core, name)
    setattr(core, name, fn)
    setattr(oracle, name, fn)
    try:
        yield
    finally:
        setattr(core, name, old)
        setattr(oracle, name, old)


def pin_functions():
    return [f for n, f in inspect.getmembers(pins, inspect.isfunction)
            if n.startswith("test_") and not inspect.signature(f).parameters]


def caught(name, fn):
    """True if at least one pin's assertion fails with the mutant in place
    (an error of another kind would not show that the pin checks anything)."""
    with patched(name, fn):
        for f in pin_functions():
            try:
                with np.errstate(all="ignore"):
                    f()
            except AssertionError:
                return True
    return False


_orig = {n: getattr(core, n) for n in dir(core) if not n.startswith("_")}


def _logits_over_d(q, K):
    return (K @ q) / K.shape[-1]


def _decode_drop_logc(q, Km, Vm, Kr, Vr, logc, cfg, return_stats=False):
    return _orig["shared_softmax_decode"](q, Km, Vm, Kr, Vr, np.zeros_like(logc), cfg, return_stats)


def _gate_wrong_sign(p_max, tau, alpha, g_min):
    return max(g_min, core.sigmoid(alpha * (p_max - tau)))


def _gate_temperature(p_max, tau, alpha, g_min):
    return max(g_min, core.sigmoid((tau - p_max) / alpha))


def _decode_residual_numerator_only(q, Km, Vm, Kr, Vr, logc, cfg, return_stats=False):
    a = core.logits(q, Km)
    mu = a.max()
    e = np.exp(a - mu)
    p_max = 1.0 / e.sum()
    g = core.dynamic_gate(p_max, cfg.tau, cfg.alpha, cfg.g_min) if cfg.gate_mode == 0 else cfg.g_fixed
    at = core.logits(q, Kr) + logc + (np.log(g) if g > 0 else -np.inf) if Kr.shape[0] else np.zeros(0)
    wr = np.exp(at - mu)
    out = (e @ Vm + (wr @ Vr if Kr.shape[0] else 0.0)) / e.sum()       # Z^ misses the residual
    if return_stats:
        return out, dict(p_max=p_max, g=g, Z=e.sum(), N=e @ Vm, shift=mu)
    return out


def _decode_gate_on_main(q, Km, Vm, Kr, Vr, logc, cfg, return_stats=False):
    # the gate applied to the main branch instead of the residual one
    a = core.logits(q, Km)
    mu = a.max()
    p_max = 1.0 / np.exp(a - mu).sum()
    g = core.dynamic_gate(p_max, cfg.tau, cfg.alpha, cfg.g_min) if cfg.gate_mode == 0 else cfg.g_fixed
    lg = np.log(g) if g > 0 else -np.inf
    at = core.logits(q, Kr) + logc if Kr.shape[0] else np.zeros(0)
    allv = np.concatenate([a + lg, at])
    m = np.max(allv[np.isfinite(allv)])
    w = np.exp(allv - m)
    V = np.concatenate([Vm, Vr]) if Kr.shape[0] else Vm
    out = (w @ V) / w.sum()
    if return_stats:
        return out, dict(p_max=p_max, g=g, Z=w.sum(), N=w @ V, shift=m)
    return out


def _scores_no_head_average(K, Qfit, pool):
    return _orig["scores_obs_pool"](K, Qfit, pool) * Qfit.shape[0]


def _scores_edge_normalised(K, Qfit, pool):
    out = _orig["scores_obs_pool"](K, Qfit, pool)
    s, h = K.shape[0], pool // 2
    n = np.array([min(p + h, s - 1) - max(p - h, 0) + 1 for p in range(s)], dtype=float)
    return out * pool / n


def _scores_no_softmax(K, Qfit, pool):
    G, n_fit, _ = Qfit.shape
    acc = np.zeros(K.shape[0])
    for g in range(G):
        for t in range(n_fit):
            acc += np.exp(core.logits(Qfit[g, t], K)) / G
    padded = np.concatenate([np.zeros(pool // 2), acc, np.zeros(pool // 2)])
    return sum(padded[j:j + K.shape[0]] for j in range(pool)) / pool


def _rank_ties_high(scores, recent):
    n = max(scores.shape[0] - recent, 0)
    pos = np.arange(n)
    return pos[np.lexsort((-pos, -scores[:n]))]


def _rank_includes_recent(scores, recent):
    return _orig["rank_evictable"](scores, 0)[: max(scores.shape[0] - recent, 0)]


def _select_off_by_one(ranked, s, recent, m):
    M, E = _orig["select_main"](ranked, s, recent, m + 1)
    return M, E


def _lloyd_init_low(K, V, E, r, iters):
    return _orig["lloyd_residual"](K, V, np.concatenate([E[r:], E[:r]]) if len(E) > r else E, r, iters)


def _lloyd_one_iteration(K, V, E, r, iters):
    return _orig["lloyd_residual"](K, V, E, r, 1)


def _assign_ties_high(KE, centers):
    d = np.sum(centers * centers, axis=1)[None, :] - 2.0 * (KE @ centers.T)
    return centers.shape[0] - 1 - np.argmin(d[:, ::-1], axis=1)


def _assign_no_norm(KE, centers):
    return np.argmax(KE @ centers.T, axis=1)


def _choose_r_non_strict(L0, rs, losses, delta):
    if len(rs) == 0:
        return 0
    i = int(np.argmin(losses))
    return rs[i] if losses[i] <= (1.0 - delta) * L0 else 0


def _choose_r_largest_on_tie(L0, rs, losses, delta):
    if len(rs) == 0:
        return 0
    order = sorted(range(len(rs)), key=lambda i: (losses[i], -rs[i]))
    best = order[0]
    return rs[best] if losses[best] < (1.0 - delta) * L0 else 0


def _round_truncate(x):
    x = np.asarray(x, dtype=np.float64)
    mant, expo = np.frexp(x)
    return np.ldexp(np.trunc(np.ldexp(mant, 8)), expo - 8)


def _logc_plus_one(counts, beta):
    return beta * np.log(counts.astype(np.float64) + 1.0)


def _keynorm_abs(K):
    return np.sum(np.abs(K), axis=1)


def _nearest_fp64(k, kbar):
    return int(np.argmin(np.sum((kbar - k) ** 2, axis=1)))


def _nearest_ties_high(k, kbar):
    d = [float(np.sum((kbar[j] - k) ** 2)) for j in range(kbar.shape[0])]
    return int(len(d) - 1 - np.argmin(d[::-1]))


def _fold_halfway(kbar_j, vbar_j, c_j, k, v, beta):
    return (orc_round((kbar_j + k) / 2), orc_round((vbar_j + v) / 2), c_j + 1,
            beta * np.log(c_j + 1.0))


def _fold_count_stays(kbar_j, vbar_j, c_j, k, v, beta):
    kb, vb, c, lc = _orig["fold_into_entry"](kbar_j, vbar_j, c_j, k, v, beta)
    return kb, vb, c_j, beta * np.log(max(c_j, 1))


def _ring_evicts_newest(cache, k_new, v_new, positions, n_app, capacity, policy, beta=1.0):
    out, na = cache, n_app
    for t in range(len(positions)):
        if na == capacity:
            if policy == core.APPEND_FAIL:
                raise ValueError("full")
            out = core.UnitCache(main_pos=out.main_pos[:-1], kmain=out.kmain[:-1],
                                 vmain=out.vmain[:-1], kbar=out.kbar, vbar=out.vbar,
                                 counts=out.counts, logc=out.logc, r=out.r)
            na -= 1
        out = core.append_tokens(out, k_new[t:t + 1], v_new[t:t + 1], positions[t:t + 1])
        na += 1
    return out, na


def orc_round(x):
    return _orig["round_to_bf16"](x)


def _keynorm_in_dim_order(K):
    acc = np.zeros(K.shape[0])
    for i in range(K.shape[1]):
        acc = acc + K[:, i] * K[:, i]
    return acc


def _val_loss_no_mean(cache, Qval, O_full, cfg):
    return _orig["validation_loss"](cache, Qval, O_full, cfg) * Qval.shape[0] * Qval.shape[1]


def _separate_additive(q, Kmain, Vmain, Kres, Vres, logc, cfg, return_stats=False):
    out, st = _orig["separate_softmax_decode"](q, Kmain, Vmain, Kres, Vres, logc, cfg, True)
    o_main = _orig["separate_softmax_decode"](q, Kmain, Vmain, Kres[:0], Vres[:0], logc[:0], cfg)
    g = st["g"]
    return o_main + (out - (1 - g) * o_main)          # o_M + g o_R instead of a mixture


def _separate_drop_logc(q, Kmain, Vmain, Kres, Vres, logc, cfg, return_stats=False):
    lc = np.where(np.isfinite(logc), 0.0, logc)
    return _orig["separate_softmax_decode"](q, Kmain, Vmain, Kres, Vres, lc, cfg, return_stats)


def _append_replaces_last_main(cache, k_new, v_new, positions):
    n = len(positions)
    return _orig["append_tokens"](orc_unit_drop_last(cache, n), k_new, v_new, positions)


def orc_unit_drop_last(cache, n):
    return core.UnitCache(main_pos=cache.main_pos[:len(cache.main_pos) - n],
                          kmain=cache.kmain[:len(cache.kmain) - n],
                          vmain=cache.vmain[:len(cache.vmain) - n], kbar=cache.kbar,
                          vbar=cache.vbar, counts=cache.counts, logc=cache.logc, r=cache.r)


def _append_as_residual(cache, k_new, v_new, positions):
    return core.UnitCache(main_pos=cache.main_pos, kmain=cache.kmain, vmain=cache.vmain,
                          kbar=np.vstack([cache.kbar, k_new]), vbar=np.vstack([cache.vbar, v_new]),
                          counts=np.concatenate([cache.counts, np.ones(len(positions), int)]),
                          logc=np.concatenate([cache.logc, np.zeros(len(positions))]),
                          r=cache.r + len(positions))


def _attention_full_no_shift(q, K, V):
    a = core.logits(q, K)
    w = np.exp(a)
    return (w @ V) / (w.sum() + 1.0)



def _adakv_generic(scores, budget, recent, safeguard, *, head_desc=False, pool_all=False,
                   f_of=None, n_of=None):
    """AdaKV allocation with one planted deviation (see the mutants below)."""
    H, s = scores.shape
    if budget >= s:
        return np.full(H, budget, dtype=np.int64)
    n_p = min(recent, s)
    n = n_of(budget, n_p) if n_of else budget - n_p
    f = f_of(safeguard, n) if f_of else int(np.floor(float(np.float32(safeguard)) * n))
    f = min(max(f, 0), n)
    sc, hd, ps = [], [], []
    for h in range(H):
        rest = core.rank_evictable(scores[h], recent)[0 if pool_all else f:]
        sc.append(scores[h][rest])
        hd.append(np.full(len(rest), h))
        ps.append(rest)
    sc, hd, ps = np.concatenate(sc), np.concatenate(hd), np.concatenate(ps)
    order = np.lexsort((ps, -hd if head_desc else hd, -sc))
    picked = hd[order[:H * (n - f)]]
    return n_p + f + np.bincount(picked, minlength=H).astype(np.int64)


def _adakv_ties_high_head(scores, budget, recent, safeguard):
    return _adakv_generic(scores, budget, recent, safeguard, head_desc=True)


def _adakv_pool_includes_safeguard(scores, budget, recent, safeguard):
    return _adakv_generic(scores, budget, recent, safeguard, pool_all=True)


def _adakv_safeguard_rounded(scores, budget, recent, safeguard):
    return _adakv_generic(scores, budget, recent, safeguard,
                          f_of=lambda sg, n: int(round(float(np.float32(sg)) * n)))


def _adakv_window_not_protected(scores, budget, recent, safeguard):
    return _adakv_generic(scores, budget, recent, safeguard, n_of=lambda b, n_p: b)


MUTANTS = [
    ("logits", _logits_over_d),
    ("shared_softmax_decode", _decode_drop_logc),
    ("shared_softmax_decode", _decode_residual_numerator_only),
    ("shared_softmax_decode", _decode_gate_on_main),
    ("dynamic_gate", _gate_wrong_sign),
    ("dynamic_gate", _gate_temperature),
    ("scores_obs_pool", _scores_no_head_average),
    ("scores_obs_pool", _scores_edge_normalised),
    ("scores_obs_pool", _scores_no_softmax),
    ("rank_evictable", _rank_ties_high),
    ("rank_evictable", _rank_includes_recent),
    ("select_main", _select_off_by_one),
    ("lloyd_residual", _lloyd_init_low),
    ("lloyd_residual", _lloyd_one_iteration),
    ("lloyd_assign", _assign_ties_high),
    ("lloyd_assign", _assign_no_norm),
    ("choose_r", _choose_r_non_strict),
    ("choose_r", _choose_r_largest_on_tie),
    ("round_to_bf16", _round_truncate),
    ("log_counts", _logc_plus_one),
    ("scores_keynorm", _keynorm_abs),
    ("scores_keynorm", _keynorm_in_dim_order),
    ("nearest_entry", _nearest_fp64),
    ("nearest_entry", _nearest_ties_high),
    ("fold_into_entry", _fold_halfway),
    ("fold_into_entry", _fold_count_stays),
    ("append_ring", _ring_evicts_newest),
    ("validation_loss", _val_loss_no_mean),
    ("attention_full", _attention_full_no_shift),
    ("separate_softmax_decode", _separate_additive),
    ("separate_softmax_decode", _separate_drop_logc),
    ("append_tokens", _append_replaces_last_main),
    ("append_tokens", _append_as_residual),
    ("adakv_budgets", _adakv_ties_high_head),
    ("adakv_budgets", _adakv_pool_includes_safeguard),
    ("adakv_budgets", _adakv_safeguard_rounded),
    ("adakv_budgets", _adakv_window_not_protected),
]


@pytest.mark.parametrize("name,fn", MUTANTS, ids=[f"{n}:{f.__name__}" for n, f in MUTANTS])
def test_pins_catch_planted_mistake(name, fn):
    assert caught(name, fn), f"no pin fails when {name} carries the mistake {fn.__name__}"


def test_unmutated_oracle_passes_every_pin():
    for f in pin_functions():
        f()
