"""Stage-wise parity checks of GPU construction against the fp64 oracle.

Protocol (float32 on the GPU, float64 in the oracle):
  scores     relative error <= 1e-4;
  ranking    bit-exact when the oracle ranks the GPU's own scores; against the
             oracle's fp64 scores, two positions may only trade places if their
             fp64 scores differ by < 1e-5 relative (a near tie);
  key-norm   scores and selection bit-exact;
  entries    given the GPU's evicted set in the GPU's rank order, the oracle's
             Lloyd gives exactly the same counts (the GPU certifies each
             nearest-centre choice in fp64) and the same bf16 entries (at most
             one ulp apart in 0.1% of the values: fp64 sums in another order);
  r choice   equal unless the oracle's deciding margin is < 1e-3 relative.
"""
import numpy as np
import torch

import oracle as orc
from paper_2607_29591_gb300 import reskv as R

from helpers import assert_output_parity, bf16_to_f64, errors, unit_from_layout

NEAR_TIE = 1e-5


def check_ranking(gpu_scores, gpu_top, ref_scores, recent, keynorm):
    """Ranking protocol for one unit; returns the number of near-tie swaps."""
    n_top = len(gpu_top)
    own = orc.rank_evictable(gpu_scores, recent)[:n_top]
    assert np.array_equal(own, gpu_top), "GPU ranking differs from ranking its own scores"
    ref = orc.rank_evictable(ref_scores, recent)[:n_top]
    if keynorm:
        assert np.array_equal(gpu_scores, ref_scores)
        assert np.array_equal(ref, gpu_top)
        return 0
    np.testing.assert_allclose(gpu_scores, ref_scores, rtol=1e-4, atol=0)
    swaps = 0
    for i in np.nonzero(ref != gpu_top)[0]:
        a, b = ref_scores[ref[i]], ref_scores[gpu_top[i]]
        assert abs(a - b) <= NEAR_TIE * max(abs(a), abs(b)), f"rank {i}: not a near tie"
        swaps += 1
    return swaps


def check_entries(gpu_unit, K, V, gpu_top, recent, s, b, iters):
    """Oracle Lloyd on the GPU's evicted set (GPU rank order) vs GPU entries."""
    r = gpu_unit.r
    if r == 0:
        return
    m = b - r
    keep = m - recent
    main = set(gpu_unit.main_pos.tolist())
    assert len(main) == m
    rest = [p for p in range(s - recent) if p not in set(gpu_top[:keep].tolist())]
    in_top = set(gpu_top.tolist())
    E = np.array(list(gpu_top[keep:]) + [p for p in rest if p not in in_top])
    assert not (set(E.tolist()) & main) and len(E) == s - m
    kbar, vbar, counts = orc.lloyd_residual(K, V, E, r, iters)
    kb, vb = orc.round_to_bf16(kbar), orc.round_to_bf16(vbar)
    # the GPU certifies every nearest-centre decision in fp64, so the
    # assignments, hence the counts, are the oracle's exactly
    assert np.array_equal(counts, gpu_unit.counts), \
        f"{int(np.sum(counts != gpu_unit.counts))} of {r} entry counts differ"
    # means: fp64 sums in different orders, then the same bf16 rounding
    for mine, ref in ((gpu_unit.kbar, kb), (gpu_unit.vbar, vb)):
        ulp = np.abs(ref) * 2.0 ** -7 + 1e-30
        assert np.all(np.abs(mine - ref) <= ulp)
        assert np.mean(mine == ref) > 0.999


def decode_parity(cache, lay, ref_units, Ks, Qd, w, ocfg_of):
    """GPU decode of the GPU-built cache vs oracle decode of the oracle cache."""
    L, Bt, H, G = w.n_layers, w.batch, w.n_kv_heads, w.group
    O = torch.empty(Qd.shape, dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(cache, -1, Qd, O)
    torch.cuda.synchronize()
    O = O.cpu().numpy()
    qf = bf16_to_f64(Qd)
    worst = 0.0
    for u, ref in ref_units.items():
        l, rem = divmod(u, Bt * H)
        b, h = divmod(rem, H)
        q = qf[l, b, h * G:(h + 1) * G]
        ref_o = orc.decode_unit(ref, q, ocfg_of(u))
        mx, rel = assert_output_parity(O[l, b, h * G:(h + 1) * G], ref_o, f"unit {u}")
        # the kernel alone: oracle decode of the GPU's own cache
        own = orc.decode_unit(unit_from_layout(lay, u), q, ocfg_of(u))
        assert errors(O[l, b, h * G:(h + 1) * G], own)[1] < 1e-4
        worst = max(worst, rel)
    return worst




# ---------------------------------------------------------------------------
# oracle construction in worker processes (full-size tests)
# ---------------------------------------------------------------------------

def stratified_units(w, n):
    """n units spread over layers, batch elements and KV heads (all units if
    the workload has at most n)."""
    if n >= w.n_units:
        return list(range(w.n_units))
    out = []
    for i in range(n):
        l = (i * w.n_layers) // n
        b = (i * 5 + i // 3) % w.batch
        h = (i * 3 + i // w.n_kv_heads) % w.n_kv_heads
        out.append((l * w.batch + b) * w.n_kv_heads + h)
    return sorted(set(out))


def input_digest(*tensors):
    import hashlib
    h = hashlib.sha256()
    for t in tensors:
        if t is not None:
            h.update(t.contiguous().view(torch.int16).numpy().tobytes())
    return h.hexdigest()


def oracle_build_job(args):
    """Worker: regenerate one unit's inputs on the CPU and run the oracle's
    Alg. 1 on them.  Returns (unit, oracle cache, digest of the inputs)."""
    from paper_2607_29591_gb300 import workloads as wl
    name, u, delta, r_override = args
    w = wl.WORKLOADS[name]
    l, rem = divmod(u, w.batch * w.n_kv_heads)
    b, h = divmod(rem, w.n_kv_heads)
    Kc, Vc = wl.unit_kv(w, l, b, h, "cpu")
    Qc = wl.unit_obs_queries(w, l, b, h, Kc, "cpu") if w.n_obs > 0 else None
    oc = orc.OracleConfig(budget=w.budget, recent_window=w.recent_window, n_fit=w.n_fit,
                          n_val=w.n_val, score_mode=w.score_mode, residual_override=r_override,
                          delta=delta)
    ref = orc.build_unit(bf16_to_f64(Kc), bf16_to_f64(Vc),
                         None if Qc is None else bf16_to_f64(Qc), oc)
    return u, ref, input_digest(Kc, Vc, Qc)


def _single_thread():
    torch.set_num_threads(1)


def oracle_pool(n_jobs):
    """Spawned worker processes (one BLAS thread each) for oracle builds."""
    import concurrent.futures
    import multiprocessing
    import os
    procs = max(1, min(n_jobs, os.cpu_count() or 1))
    old = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS",
                                          "MKL_NUM_THREADS")}
    for k in old:
        os.environ[k] = "1"
    try:
        return concurrent.futures.ProcessPoolExecutor(
            procs, mp_context=multiprocessing.get_context("spawn"), initializer=_single_thread)
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def r_margin(losses, delta):
    """The oracle's deciding margin for r: the distance of L_r*/L_0 from the
    threshold 1 - delta, and the relative gap between the two best L_r."""
    rs = sorted(k for k in losses if k > 0)
    if not rs:
        return 1.0
    best = min(rs, key=lambda r: (losses[r], r))
    margin = abs(losses[best] / losses[0] - (1 - delta)) if losses[0] > 0 else 1.0
    vals = sorted(losses[r] for r in rs)
    gap = (vals[1] - vals[0]) / vals[0] if len(vals) > 1 and vals[0] > 0 else 1.0
    return min(margin, gap)


def check_r(gu_r, ref, delta, u, skipped, margin_band=1e-3):
    """r of the GPU's unit against the oracle's, unless the oracle's deciding
    margin lies inside the band (then the unit is recorded in `skipped`)."""
    if r_margin(ref.losses, delta) <= margin_band:
        skipped.append(u)
    else:
        assert gu_r == ref.r, f"unit {u}: r {gu_r} vs oracle {ref.r}"


def assert_few_skipped(skipped, n_checked, what=""):
    """At most 5 % of the checked units (at least one allowed) may fall inside
    the margin band; the count is printed with -s / -rA."""
    print(f"{what}: r compared on {n_checked - len(skipped)} of {n_checked} units; "
          f"inside the margin band: {skipped}")
    assert len(skipped) <= max(1, int(np.ceil(0.05 * n_checked))), (what, skipped)
