"""fp64 CPU oracle for ResKV construction and shared-softmax decode.

TEST INFRASTRUCTURE ONLY.  This module is a plain, slow, obviously-correct
restatement of the paper "ResKV: Reconstructing Omitted Attention
Contributions for Fixed-Budget KV Cache Compression" in numpy float64.  Only
``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference
leg of ``bench.py`` may import it.  It shares no code with the CUDA library
(``paper_2607_29591_gb300``) and imports nothing from it; the product path
never calls it.

Every function follows one passage of the paper, named in its docstring
(section, equation label or algorithm).  Inputs arrive as bf16 values that are
upcast exactly to float64; all arithmetic is float64.  Where the paper is
silent the reading taken is stated at the function (the same list is kept in
the project's design notes):

* observation queries: the caller supplies ``n_obs`` rows per query head, the
  first ``n_fit`` are the fit part and the last ``n_val`` the validation part
  (Sec. 5.5.1), and every observation query attends to all ``s`` tokens;
* SnapKV scores: per fit query and head, softmax over all tokens; the weights
  are averaged over the GQA group and summed over fit queries, then average
  pooled with a zero-padded window of ``pool`` (5) tokens (App. B.2);
* query-free scoring (no observation window): ``s_p = ||k_p||^2`` -- a build
  choice, the paper defines no such rule -- as the exact sum of the squares
  rounded once to float64 (independent of summation order);
* ranking ties go to the lower token index; Lloyd assignment ties go to the
  lower centre index; an empty cluster keeps its centre and ends with count 0
  (log-count ``-inf``: the slot contributes nothing);
* candidate budgets ``r = floor(ratio * b)`` over the ratio grid, duplicates
  and zero dropped; ``argmin`` ties go to the smaller ``r``; the residual is
  enabled only on a strict improvement (Eq. valproxy);
* stored residual entries are rounded to bf16 (round-to-nearest-even); the
  validation loss is evaluated on the stored (rounded) entries;
* the validation loss averages over validation queries and the G query heads
  of the KV head;
* decode-time growth into a bounded region of appended tokens: once it is
  full, the oldest appended token leaves the exact window and is dropped or
  folded into its nearest residual entry (exact squared distance, ties to the
  lower entry) as a running mean (c k_bar + k) / (c + 1) in float64, stored as
  bf16, count + 1;
* AdaKV budgets (App. B, "AdaKV": SnapKV scores, safeguard 0.2): the KV heads
  of one (layer, batch element) share H*b slots; every head keeps its window
  P and its own f = floor(safeguard * (b - |P|)) best tokens, and the other
  H*(b - |P| - f) slots go to the best-scored remaining tokens of all heads
  (ties: lower head, then lower position); each head is then built by Alg. 1
  with its own budget b_h.

Parity status: every function here is pinned by ``tests/test_oracle_pins.py``
against closed forms, fixed points or hand-computed fixtures; none is
"parity unpinned".  The end-to-end accuracy numbers of the paper (RULER,
LongBench) are not reproducible here (no model weights or benchmark data).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import Optional, Sequence

import numpy as np

# ---------------------------------------------------------------------------
# Hyper-parameters (App. B, "ResKV Construction Settings")
# ---------------------------------------------------------------------------

GATE_DYNAMIC = 0
GATE_FIXED = 1

SCORE_OBS_POOL = 0
SCORE_KEYNORM = 1

SOFTMAX_SHARED = 0        # Eq. reskv: one softmax over main and residual entries
SOFTMAX_SEPARATE = 1      # "w/o shared softmax" ablation (Table ablation_main)


@dataclass
class OracleConfig:
    """Construction / decode settings for one (layer, KV head) unit.

    Defaults are the paper's (App. B "ResKV Construction Settings"; App. B.2
    SnapKV: window protection 64, pooling kernel 5).
    """

    budget: int                      # b, slots per (layer, KV head)   (Sec. 3.2)
    recent_window: int = 64          # |P|, protected recent tokens   (Eq. main_selection)
    n_fit: int = 96                  # fitting queries                 (Sec. 5.5.1)
    n_val: int = 32                  # validation queries              (Sec. 5.5.1)
    pool_kernel: int = 5             # SnapKV average pooling          (App. B.2)
    score_mode: int = SCORE_OBS_POOL
    grid_ratios: Sequence[float] = (0.0, 0.05, 0.10, 0.15, 0.20)  # App. B
    lloyd_iters: int = 4             # App. B
    delta: float = 0.01              # Eq. valproxy margin
    beta: float = 1.0                # count exponent in the residual logit (App. B)
    residual_override: Optional[int] = None  # fixed r, bypasses the proxy
    gate_mode: int = GATE_DYNAMIC
    tau: float = 0.25                # Eq. gate threshold (App. B)
    alpha: float = 12.0              # sigmoid slope = 1/T_g (App. B)
    g_min: float = 0.0               # minimum gate (App. B)
    g_fixed: float = 1.0             # gate value when gate_mode == GATE_FIXED
    softmax_mode: int = SOFTMAX_SHARED


# ---------------------------------------------------------------------------
# bf16 helpers (storage format of the cache; not part of the method)
# ---------------------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact upcast of bf16 bit patterns (uint16) to float64."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bf16 value, ties to even.

    bf16 keeps 8 significant bits down to 2^-126; below that (subnormals) its
    spacing stays 2^-133.  Each value is divided by the spacing at its
    magnitude (a power of two: exact), rounded to an integer (numpy rint:
    half to even) and scaled back, so no float32 double rounding occurs.
    Zero stays zero; values beyond the bf16 range are not expected here.
    """
    x = np.asarray(x, dtype=np.float64)
    _, expo = np.frexp(x)                    # |x| in [2^(expo-1), 2^expo)
    quantum = np.maximum(expo - 8, -133)     # exponent of the spacing at |x|
    return np.ldexp(np.rint(np.ldexp(x, -quantum)), quantum)


# ---------------------------------------------------------------------------
# Attention statistics (Sec. 3.1, Sec. 4.2)
# ---------------------------------------------------------------------------

def logits(q: np.ndarray, K: np.ndarray) -> np.ndarray:
    """a_p(q) = <q, k_p> / sqrt(d)  (Sec. 4.1, Eq. expand; Sec. 5.4)."""
    d = K.shape[-1]
    return (K @ q) / np.sqrt(d)


def attention_full(q: np.ndarray, K: np.ndarray, V: np.ndarray) -> np.ndarray:
    """o_S(q) = softmax(q K^T / sqrt(d)) V over all rows  (Eq. attn)."""
    a = logits(q, K)
    w = np.exp(a - a.max())
    return (w @ V) / w.sum()


def zn_stats(q: np.ndarray, K: np.ndarray, V: np.ndarray, shift: float = 0.0):
    """Unnormalised statistics Z_T(q), N_T(q) of a token set  (Eq. zn).

    Returned as e^{-shift} Z and e^{-shift} N so that callers can keep a common
    scale between several sets without overflow.
    """
    a = logits(q, K)
    e = np.exp(a - shift)
    return e.sum(), e @ V


# ---------------------------------------------------------------------------
# Token scoring (App. B.2 SnapKV rule; Alg. 1)
# ---------------------------------------------------------------------------

def scores_obs_pool(K: np.ndarray, Qfit: np.ndarray, pool: int) -> np.ndarray:
    """SnapKV-style token scores from the fit observation queries.

    ``K``: [s, d]; ``Qfit``: [G, n_fit, d] (the fit rows of the G query heads
    that share this KV head).  For every fit query and head the attention
    weights over all s tokens are formed; they are averaged over the G heads
    (GQA: one score per KV head, App. B) and summed over fit queries; the sum
    is average pooled with a zero-padded window of ``pool`` tokens.
    """
    G, n_fit, d = Qfit.shape
    s = K.shape[0]
    if pool < 1 or pool % 2 == 0:
        raise ValueError("pool kernel must be a positive odd integer")
    acc = np.zeros(s, dtype=np.float64)
    for g in range(G):
        for t in range(n_fit):
            a = logits(Qfit[g, t], K)
            w = np.exp(a - a.max())
            acc += (w / w.sum()) / G
    half = pool // 2
    padded = np.concatenate([np.zeros(half), acc, np.zeros(half)])
    pooled = np.zeros(s, dtype=np.float64)
    for j in range(pool):                      # (A_{p-h} + ... + A_{p+h}) / pool
        pooled += padded[j:j + s]
    return pooled / pool


def scores_keynorm(K: np.ndarray) -> np.ndarray:
    """Query-free score s_p = ||k_p||^2 (a build choice; the paper has none):
    the exact sum of the squares, rounded once to float64.

    Every square of a bf16 value is exact in float64 (8 significant bits
    squared), so math.fsum, which returns the correctly rounded sum of its
    exact inputs, gives the exact score whatever the order of the dims."""
    return np.array([math.fsum(row) for row in K * K], dtype=np.float64)


# ---------------------------------------------------------------------------
# Main-cache selection (Sec. 5.2, Eq. main_selection)
# ---------------------------------------------------------------------------

def rank_evictable(scores: np.ndarray, recent: int) -> np.ndarray:
    """Positions of S \\ P ordered by score, highest first; ties -> lower index.

    P is the protected window of the last ``recent`` positions.
    """
    s = scores.shape[0]
    n = max(s - recent, 0)
    pos = np.arange(n)
    # lexsort sorts by the last key first: primary = -score, secondary = index
    order = np.lexsort((pos, -scores[:n]))
    return pos[order]


def select_main(ranked: np.ndarray, s: int, recent: int, m: int):
    """M = P u Top_{m-|P|}(s), E = S \\ M  (Eq. main_selection).

    Returns (M as ascending positions, E in rank order).  E in rank order is
    what Lloyd initialisation needs (App. B: initial centres are the evicted
    keys with the highest scores).
    """
    n_p = min(recent, s)
    take = m - n_p
    if take < 0:
        raise ValueError("main budget smaller than the protected window")
    P = np.arange(s - n_p, s)
    top = ranked[:take]
    M = np.sort(np.concatenate([top, P]))
    E = ranked[take:]
    return M, E


def candidate_budgets(budget: int, ratios: Sequence[float]) -> list:
    """Residual candidates r = floor(ratio * b) > 0, distinct, ascending (App. B)."""
    rs = set()
    for ratio in ratios:
        r = int(np.floor(float(np.float32(ratio)) * budget))
        if r > 0:
            rs.add(r)
    return sorted(rs)


def adakv_budgets(scores: np.ndarray, budget: int, recent: int, safeguard: float) -> np.ndarray:
    """Per-head budgets b_h of one (layer, batch element) under AdaKV's
    allocation across KV heads (App. B, "AdaKV": SnapKV token scores, safeguard
    coefficient 0.2).

    ``scores``: [H, s], one row per KV head.  The paper gives no formula; the
    reading taken: the H heads share H*b slots.  Every head keeps its protected
    window P (Eq. main_selection) and, as the safeguard, its own
    f = floor(safeguard * (b - |P|)) highest-ranked tokens.  The remaining
    H*(b - |P| - f) slots go to the highest scores among all heads' other
    evictable tokens, ordered by score (descending), then head index, then
    position.  b_h = |P| + f + (tokens of head h in that pick).  Within a head
    the pick is a prefix of its ranking, so head h keeps exactly its top
    b_h - |P| ranked tokens, the main selection of Alg. 1 with budget b_h.
    With b >= s nothing is evicted and every head keeps b.
    """
    H, s = scores.shape
    if budget >= s:
        return np.full(H, budget, dtype=np.int64)
    n_p = min(recent, s)
    n = budget - n_p
    if n < 0:
        raise ValueError("budget smaller than the protected window")
    f = int(np.floor(float(np.float32(safeguard)) * n))
    f = min(max(f, 0), n)
    # every head's evictable tokens beyond its safeguard, as (score, head, position)
    sc, hd, ps = [], [], []
    for h in range(H):
        rest = rank_evictable(scores[h], recent)[f:]
        sc.append(scores[h][rest])
        hd.append(np.full(len(rest), h))
        ps.append(rest)
    sc, hd, ps = np.concatenate(sc), np.concatenate(hd), np.concatenate(ps)
    order = np.lexsort((ps, hd, -sc))           # score desc, then head, then position
    picked = hd[order[:H * (n - f)]]
    return n_p + f + np.bincount(picked, minlength=H).astype(np.int64)


def unit_scores(K: np.ndarray, Qobs: Optional[np.ndarray], cfg: "OracleConfig") -> np.ndarray:
    """Token scores of one unit under cfg's score mode (Alg. 1, scoring step)."""
    if cfg.score_mode == SCORE_OBS_POOL:
        return scores_obs_pool(K, Qobs[:, :cfg.n_fit], cfg.pool_kernel)
    if cfg.score_mode == SCORE_KEYNORM:
        return scores_keynorm(K)
    raise ValueError("unknown score mode")


# ---------------------------------------------------------------------------
# Residual construction (Sec. 5.3, Eq. summary, Eq. residual_partition)
# ---------------------------------------------------------------------------

def lloyd_assign(KE: np.ndarray, centers: np.ndarray) -> np.ndarray:
    """argmin_j ||k_p - c_j||^2 for every row of KE; ties -> lowest j.

    The squared distance is evaluated as ||c_j||^2 - 2<k_p, c_j> (+ ||k_p||^2,
    the same for every j and omitted) with one float64 matrix product.  A
    centre that is bit-identical to an earlier one can never win (exact ties
    go to the lower index), so such duplicates are excluded explicitly.
    """
    cn = np.sum(centers * centers, axis=1)
    dist = cn[None, :] - 2.0 * (KE @ centers.T)
    r = centers.shape[0]
    if r > 1:
        _, first = np.unique(centers, axis=0, return_index=True)
        dup = np.ones(r, dtype=bool)
        dup[first] = False
        if dup.any():
            dist[:, dup] = np.inf
    return np.argmin(dist, axis=1)             # first minimum = lowest index


def lloyd_residual(K: np.ndarray, V: np.ndarray, E: np.ndarray, r: int, iters: int):
    """Residual entries of E by Lloyd's algorithm (Sec. 5.3; App. B).

    ``E`` lists the evicted positions in rank order; the initial centres are
    the keys of its first ``r`` entries (the highest-scored evicted tokens).
    ``iters`` rounds of (assign every evicted key to its nearest centre, move
    each non-empty centre to the mean of its members).  An empty cluster keeps
    its centre.  Returns the unrounded entries (k_bar, v_bar, c) of Eq. summary
    for the final assignment: k_bar_j = mean key, v_bar_j = mean value,
    c_j = member count.
    """
    if r <= 0:
        d = K.shape[1]
        return np.zeros((0, d)), np.zeros((0, V.shape[1])), np.zeros(0, dtype=np.int64)
    if E.shape[0] < r:
        raise ValueError("fewer evicted tokens than residual entries")
    if iters < 1:
        raise ValueError("at least one Lloyd iteration is required")
    KE = K[E]
    VE = V[E]
    centers = KE[:r].copy()
    for _ in range(iters):
        assign = lloyd_assign(KE, centers)
        for j in range(r):
            members = assign == j
            if members.any():
                centers[j] = KE[members].mean(axis=0)
    counts = np.bincount(assign, minlength=r).astype(np.int64)
    vbar = np.zeros((r, V.shape[1]))
    for j in range(r):
        members = assign == j
        if members.any():
            vbar[j] = VE[members].mean(axis=0)
    return centers, vbar, counts


def log_counts(counts: np.ndarray, beta: float) -> np.ndarray:
    """beta * log c_j, with log 0 = -inf (an empty entry carries no mass)."""
    out = np.full(counts.shape, -np.inf)
    nz = counts > 0
    out[nz] = beta * np.log(counts[nz].astype(np.float64))
    return out


# ---------------------------------------------------------------------------
# Dynamic gate (Sec. 5.5.2, Eq. gate) and shared-softmax decode (Sec. 5.4)
# ---------------------------------------------------------------------------

def sigmoid(x: float) -> float:
    return 1.0 / (1.0 + np.exp(-x))


def dynamic_gate(p_max: float, tau: float, alpha: float, g_min: float) -> float:
    """g = max(g_min, sigmoid((tau - p_max) / T_g)) with T_g = 1/alpha (Eq. gate)."""
    return max(g_min, sigmoid(alpha * (tau - p_max)))


def shared_softmax_decode(q, Kmain, Vmain, Kres, Vres, logc, cfg: OracleConfig,
                          return_stats: bool = False):
    """One decode query of one query head (Alg. 2; Eqs. residual_logit, reskv_den,
    reskv_num, reskv; Eq. gate).

    a_p = <q,k_p>/sqrt(d) over the main cache; p_max = max_p softmax_M(a)_p;
    g = gate(p_max); residual logits a~_j = <q, k_bar_j>/sqrt(d) + log c_j + log g;
    Z^ = sum_M e^{a_p} + sum_R e^{a~_j};  N^ = sum_M e^{a_p} v_p + sum_R e^{a~_j} v_bar_j;
    o^ = N^ / Z^.  With R empty (or g = 0) this is eviction attention (Eq. evict).
    """
    a = logits(q, Kmain)
    mu_m = a.max()
    e_main = np.exp(a - mu_m)
    p_max = 1.0 / e_main.sum()                 # largest main-only weight: e^0 / sum
    if cfg.gate_mode == GATE_DYNAMIC:
        g = dynamic_gate(p_max, cfg.tau, cfg.alpha, cfg.g_min)
    else:
        g = cfg.g_fixed
    log_g = np.log(g) if g > 0 else -np.inf
    if Kres.shape[0] > 0:
        at = logits(q, Kres) + logc + log_g
    else:
        at = np.zeros(0)
    finite = at[np.isfinite(at)]
    mu = max(mu_m, finite.max()) if finite.size else mu_m
    w_main = np.exp(a - mu)
    w_res = np.exp(at - mu)                    # -inf logits (c = 0 or g = 0) give 0
    Z = w_main.sum() + w_res.sum()
    N = w_main @ Vmain + (w_res @ Vres if Kres.shape[0] > 0 else 0.0)
    out = N / Z
    if return_stats:
        return out, dict(p_max=p_max, g=g, Z=Z, N=N, shift=mu)
    return out


def separate_softmax_decode(q, Kmain, Vmain, Kres, Vres, logc, cfg: OracleConfig,
                            return_stats: bool = False):
    """One decode query with separate main and residual normalisations, the
    "w/o shared softmax" ablation (Sec. 6 ablation study, Table ablation_main).

    The paper names the variant but prints no combination rule; the reading
    taken here keeps every other part of the method and mixes the two
    normalised branches with the gate:

      o_M = sum_M softmax_M(a)_p v_p,          a_p = <q,k_p>/sqrt(d)
      o_R = sum_R softmax_R(a')_j v_bar_j,     a'_j = <q,k_bar_j>/sqrt(d) + log c_j
      o^  = (1 - g) o_M + g o_R,               g = gate(p_max) as in Eq. gate

    Without residual mass (R empty or every c_j = 0) or with g = 0, o^ = o_M.
    """
    a = logits(q, Kmain)
    e_main = np.exp(a - a.max())
    Z_M = e_main.sum()
    p_max = 1.0 / Z_M
    if cfg.gate_mode == GATE_DYNAMIC:
        g = dynamic_gate(p_max, cfg.tau, cfg.alpha, cfg.g_min)
    else:
        g = cfg.g_fixed
    o_main = (e_main @ Vmain) / Z_M
    ar = logits(q, Kres) + logc if Kres.shape[0] > 0 else np.zeros(0)
    finite = ar[np.isfinite(ar)]
    if finite.size == 0 or g == 0:
        out = o_main
    else:
        e_res = np.exp(ar - finite.max())      # log c_j = -inf (c = 0) gives 0
        o_res = (e_res @ Vres) / e_res.sum()
        out = (1.0 - g) * o_main + g * o_res
    if return_stats:
        return out, dict(p_max=p_max, g=g)
    return out


def decode_query(q, Kmain, Vmain, Kres, Vres, logc, cfg: OracleConfig):
    """The decode rule that cfg selects: Eq. reskv (shared softmax, the method)
    or the separate-normalisation ablation."""
    if cfg.softmax_mode == SOFTMAX_SEPARATE:
        return separate_softmax_decode(q, Kmain, Vmain, Kres, Vres, logc, cfg)
    return shared_softmax_decode(q, Kmain, Vmain, Kres, Vres, logc, cfg)


# ---------------------------------------------------------------------------
# Construction (Alg. 1) with the validation proxy (Sec. 5.5.1)
# ---------------------------------------------------------------------------

@dataclass
class UnitCache:
    """The compressed cache of one (layer, KV head) unit."""

    main_pos: np.ndarray          # [m] ascending original positions
    kmain: np.ndarray             # [m, d] exact keys
    vmain: np.ndarray             # [m, d] exact values
    kbar: np.ndarray              # [r, d] stored (bf16-rounded) mean keys
    vbar: np.ndarray              # [r, d] stored (bf16-rounded) mean values
    counts: np.ndarray            # [r] populations c_j
    logc: np.ndarray              # [r] beta * log c_j
    r: int
    # diagnostics for tests
    scores: Optional[np.ndarray] = None
    ranked: Optional[np.ndarray] = None
    losses: dict = field(default_factory=dict)
    init_order: Optional[np.ndarray] = None   # E of the chosen r in rank order


def build_candidate(K, V, ranked, cfg: OracleConfig, r: int) -> UnitCache:
    """Main cache M_r and residual entries for one candidate r (Alg. 1, candidate loop)."""
    s = K.shape[0]
    m = min(cfg.budget - r, s)
    if r == 0:
        m = min(cfg.budget, s)
    M, E = select_main(ranked, s, cfg.recent_window, m)
    kbar, vbar, counts = lloyd_residual(K, V, E, r, cfg.lloyd_iters)
    kbar_s = round_to_bf16(kbar)
    vbar_s = round_to_bf16(vbar)
    return UnitCache(main_pos=M, kmain=K[M], vmain=V[M], kbar=kbar_s, vbar=vbar_s,
                     counts=counts, logc=log_counts(counts, cfg.beta), r=r,
                     init_order=E)


def candidate_valid(s: int, cfg: OracleConfig, r: int) -> bool:
    """A candidate needs room for P in the main cache and r evicted tokens."""
    m = cfg.budget - r
    if m < min(cfg.recent_window, s):
        return False
    n_evicted = s - m
    return r <= n_evicted


def append_tokens(cache: UnitCache, k_new: np.ndarray, v_new: np.ndarray,
                  positions: np.ndarray) -> UnitCache:
    """Decode-time growth (Sec. 3.1: each decode step appends the new token's
    key and value): the new tokens join the exact main cache M, so every later
    decode attends to them exactly and counts them in p_max of the gate.  The
    residual entries stay as built (no refresh)."""
    return UnitCache(main_pos=np.concatenate([cache.main_pos, positions]),
                     kmain=np.vstack([cache.kmain, k_new]), vmain=np.vstack([cache.vmain, v_new]),
                     kbar=cache.kbar, vbar=cache.vbar, counts=cache.counts, logc=cache.logc,
                     r=cache.r, losses=cache.losses, scores=cache.scores)


# policies for a token leaving a full append region (decode-time growth)
APPEND_FAIL = 0          # no room: the append is refused
APPEND_RING_DROP = 1     # the oldest appended token leaves the cache
APPEND_RING_FOLD = 2     # the oldest appended token joins its nearest residual entry


def nearest_entry(k: np.ndarray, kbar: np.ndarray) -> int:
    """argmin_j ||k - kbar_j||^2 over the stored entries, ties -> lowest j
    (the assignment rule of Eq. residual_partition), decided exactly.

    Every bf16 value is an integer multiple of 2^-133 (the smallest bf16
    subnormal), so the squared distances are compared as exact integers after
    scaling by 2^133 (the scaling is a power of two: exact in float64)."""
    scale = 2.0 ** 133
    ki = [int(x * scale) for x in k]
    best, best_d = -1, None
    for j in range(kbar.shape[0]):
        d = sum((a - int(b * scale)) ** 2 for a, b in zip(ki, kbar[j]))
        if best_d is None or d < best_d:
            best, best_d = j, d
    return best


def fold_into_entry(kbar_j, vbar_j, c_j: int, k, v, beta: float):
    """One more member for entry j (Eq. summary as a running mean): with c_j
    members summarised by the stored means, the new means are
    (c_j kbar_j + k) / (c_j + 1) and (c_j vbar_j + v) / (c_j + 1), evaluated in
    float64 in that order and stored as bf16 (round to nearest even); the
    count becomes c_j + 1 and the logit term beta * log(c_j + 1).  An empty
    entry (c_j = 0) becomes the token itself."""
    c = float(c_j)
    kb = round_to_bf16((c * kbar_j + k) / (c + 1.0))
    vb = round_to_bf16((c * vbar_j + v) / (c + 1.0))
    return kb, vb, c_j + 1, beta * np.log(c + 1.0)


def append_ring(cache: UnitCache, k_new: np.ndarray, v_new: np.ndarray, positions: np.ndarray,
                n_app: int, capacity: int, policy: int, beta: float = 1.0):
    """Decode-time growth (Sec. 3.1: each decode step appends the new token)
    into a bounded region of `capacity` appended tokens; n_app of them are the
    last rows of the unit's main cache now.

    While the region has room the token is appended (append_tokens).  When it
    is full the oldest appended token leaves the exact window first: with
    APPEND_RING_DROP it leaves the cache; with APPEND_RING_FOLD it becomes a
    member of its nearest residual entry (nearest_entry, fold_into_entry) --
    the residual refresh that the paper leaves to future work (App. E), in the
    running-mean form of Eq. summary -- or leaves the cache when the unit has no
    residual entries.  APPEND_FAIL refuses (ValueError).  Returns the grown
    cache and its count of appended tokens."""
    out = UnitCache(main_pos=cache.main_pos.copy(), kmain=cache.kmain.copy(),
                    vmain=cache.vmain.copy(), kbar=cache.kbar.copy(), vbar=cache.vbar.copy(),
                    counts=cache.counts.copy(), logc=cache.logc.copy(), r=cache.r,
                    losses=cache.losses, scores=cache.scores)
    for t in range(len(positions)):
        if n_app == capacity:
            if policy == APPEND_FAIL or capacity == 0:
                raise ValueError("the append region is full")
            o = out.kmain.shape[0] - n_app            # the oldest appended row
            k_old, v_old = out.kmain[o].copy(), out.vmain[o].copy()
            keep = np.arange(out.kmain.shape[0]) != o
            out.kmain, out.vmain, out.main_pos = out.kmain[keep], out.vmain[keep], out.main_pos[keep]
            n_app -= 1
            if policy == APPEND_RING_FOLD and out.r > 0:
                j = nearest_entry(k_old, out.kbar)
                out.kbar[j], out.vbar[j], out.counts[j], out.logc[j] = fold_into_entry(
                    out.kbar[j], out.vbar[j], int(out.counts[j]), k_old, v_old, beta)
        out.kmain = np.vstack([out.kmain, k_new[t][None]])
        out.vmain = np.vstack([out.vmain, v_new[t][None]])
        out.main_pos = np.concatenate([out.main_pos, positions[t:t + 1]])
        n_app += 1
    return out, n_app


def decode_unit(cache: UnitCache, Q: np.ndarray, cfg: OracleConfig) -> np.ndarray:
    """Decode the G query heads of one KV head (GQA sharing, App. B): [G, d]."""
    return np.stack([decode_query(q, cache.kmain, cache.vmain, cache.kbar, cache.vbar,
                                  cache.logc, cfg) for q in Q])


def validation_loss(cache: UnitCache, Qval: np.ndarray, O_full: np.ndarray,
                    cfg: OracleConfig) -> float:
    """L_r = mean over validation queries (and the G heads) of ||o^(r) - o_S||^2
    (Eq. valloss), with the decode rule of Sec. 5.4 including the gate (or the
    ablation's rule, when cfg selects it)."""
    G, n_val, _ = Qval.shape
    total = 0.0
    for g in range(G):
        for t in range(n_val):
            o = decode_query(Qval[g, t], cache.kmain, cache.vmain, cache.kbar, cache.vbar,
                             cache.logc, cfg)
            diff = o - O_full[g, t]
            total += float(diff @ diff)
    return total / (G * n_val)


def choose_r(L0: float, rs: Sequence[int], losses: Sequence[float], delta: float) -> int:
    """r* = argmin_{r>0} L_r (ties -> smaller r); keep r* only if
    L_{r*} < (1 - delta) L_0, else r = 0  (Eq. valproxy; Alg. 1, choice of r)."""
    if len(rs) == 0:
        return 0
    order = sorted(range(len(rs)), key=lambda i: (losses[i], rs[i]))
    best = order[0]
    return rs[best] if losses[best] < (1.0 - delta) * L0 else 0


def build_unit(K: np.ndarray, V: np.ndarray, Qobs: Optional[np.ndarray],
               cfg: OracleConfig) -> UnitCache:
    """Alg. 1 for one (layer, KV head).

    ``K``, ``V``: [s, d] float64 (exact bf16 values).  ``Qobs``: [G, n_obs, d]
    observation queries of the G query heads (fit rows first), or None with the
    query-free score.
    """
    s = K.shape[0]
    # token scores on the fit queries; recent protection P
    scores = unit_scores(K, Qobs, cfg)
    ranked = rank_evictable(scores, cfg.recent_window)

    if cfg.budget >= s:                        # the budget covers every token: M = S
        out = build_candidate(K, V, ranked, cfg, 0)
        out.scores, out.ranked = scores, ranked
        return out

    if cfg.residual_override is not None:      # fixed r: the proxy is bypassed
        r = int(cfg.residual_override)
        if r > 0 and not candidate_valid(s, cfg, r):
            raise ValueError("residual override does not fit the budget")
        out = build_candidate(K, V, ranked, cfg, r)
        out.scores, out.ranked = scores, ranked
        return out

    # validation part of the observation window; its full-cache outputs
    Qval = Qobs[:, Qobs.shape[1] - cfg.n_val:]
    G = Qval.shape[0]
    O_full = np.stack([np.stack([attention_full(Qval[g, t], K, V)
                                 for t in range(cfg.n_val)]) for g in range(G)])
    # pure-main cache and L_0
    c0 = build_candidate(K, V, ranked, cfg, 0)
    L0 = validation_loss(c0, Qval, O_full, cfg)
    losses = {0: L0}
    # Alg. 1, candidate loop: every candidate r > 0
    rs = [r for r in candidate_budgets(cfg.budget, cfg.grid_ratios) if candidate_valid(s, cfg, r)]
    built = {}
    for r in rs:
        built[r] = build_candidate(K, V, ranked, cfg, r)
        losses[r] = validation_loss(built[r], Qval, O_full, cfg)
    # Alg. 1: r* and the margin test, then the cache for the chosen r
    r_star = choose_r(L0, rs, [losses[r] for r in rs], cfg.delta)
    out = built[r_star] if r_star > 0 else c0
    out.scores, out.ranked, out.losses = scores, ranked, losses
    return out


def build_heads_adakv(Ks: np.ndarray, Vs: np.ndarray, Qobs: Optional[np.ndarray],
                      cfgs: Sequence["OracleConfig"], safeguard: float):
    """AdaKV allocation across the H KV heads of one (layer, batch element),
    then Alg. 1 for every head with its own budget (App. B, "AdaKV" with
    ResKV on top: Table ruler_paper, Table longbench_paper "+ResKV" rows).

    ``Ks``, ``Vs``: [H, s, d]; ``Qobs``: [H, G, n_obs, d] or None; ``cfgs``: one
    OracleConfig per head carrying the shared budget b (they may differ in
    residual_override).  Returns (budgets [H], list of UnitCache).
    """
    H = Ks.shape[0]
    scores = np.stack([unit_scores(Ks[h], None if Qobs is None else Qobs[h], cfgs[h])
                       for h in range(H)])
    budgets = adakv_budgets(scores, cfgs[0].budget, cfgs[0].recent_window, safeguard)
    units = [build_unit(Ks[h], Vs[h], None if Qobs is None else Qobs[h],
                        replace(cfgs[h], budget=int(budgets[h]))) for h in range(H)]
    return budgets, units
