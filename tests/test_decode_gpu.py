"""GPU decode (Alg. 2) through the C ABI against the fp64 oracle.

Caches are imported through reskv_import_cache: either built by the oracle
(Alg. 1 in fp64) or assembled from seeded synthetic rows with ragged
main/residual splits, so that the decode kernel is checked on its own.
"""
import math

import numpy as np
import pytest
import torch
from scipy.special import softmax

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R
from paper_2607_29591_gb300 import workloads as wl

from helpers import (assert_output_parity, bf16_bits, bf16_to_f64, empty_layout, errors,
                     put_unit, unit_from_layout)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


KERNEL = {"id": R.RESKV_DECODE_MMA}
# Launches that cut units differently agree to fp32 rounding, not bit for bit:
# every warp's piece raises its softmax reference maxima on its own tiles, so
# the weights are scaled (and split into bf16 hi + lo parts) differently.
SPLIT_REL = 1e-5


@pytest.fixture(autouse=True, params=[R.RESKV_DECODE_FMA, R.RESKV_DECODE_MMA, R.RESKV_DECODE_CLUSTER,
                                      R.RESKV_DECODE_LSE_MERGE],
                ids=["fma", "mma", "cluster", "lse"])
def decode_kernel(request):
    """Every decode test runs on the four decode paths: CUDA-core FMA,
    tensor-core stream-K, tensor-core one-cluster-per-unit, and the paper-style
    comparison path (branch passes merged through log-sum-exp statistics)."""
    KERNEL["id"] = request.param
    yield request.param


def mkcfg(**kw):
    return R.reskv_config_default(decode_kernel=KERNEL["id"], **kw)


def ocfg_from(cfg):
    return orc.OracleConfig(budget=cfg.budget, gate_mode=cfg.gate_mode, tau=cfg.tau,
                            alpha=cfg.alpha, g_min=cfg.g_min, g_fixed=cfg.g_fixed,
                            softmax_mode=cfg.softmax_mode)


def synthetic_layout(L, Bt, H, b, splits, seed_layer=0, s=None):
    """Units filled with generator rows: main = first m rows, residual = next r
    rows, counts drawn from the hash (some zero)."""
    U = L * Bt * H
    s = s or (b + 64)
    w = wl.Workload("synthetic", L, Bt, H, 4, 128, s, b, 0, 0, 0, 0, "fixed:0", 1)
    lay = empty_layout(U, b)
    rng = np.random.default_rng(1234)
    for u in range(U):
        m, r = splits[u]
        l, rem = divmod(u, Bt * H)
        bb, h = divmod(rem, H)
        K, V = wl.unit_kv(w, l + seed_layer, bb, h)
        lay["n_main"][u], lay["n_res"][u] = m, r
        lay["kslots"][u, :m + r] = bf16_bits(K[:m + r])
        lay["vslots"][u, :m + r] = bf16_bits(V[:m + r])
        lay["slot_pos"][u, :m] = np.arange(m)
        if r:
            c = rng.integers(0, 200, r)
            c[rng.random(r) < 0.1] = 0
            lay["counts"][u, m:m + r] = c
            with np.errstate(divide="ignore"):
                lay["logc"][u, m:m + r] = np.log(c.astype(np.float64)).astype(np.float32)
    return w, lay


def queries_for(w, L, Bt, H, G, lay_K_source_rows=None, step=0):
    """Decode queries [L, B, H*G, d] aimed at the units' first rows."""
    Q = torch.empty((L, Bt, H * G, 128), dtype=torch.bfloat16)
    for l in range(L):
        for bb in range(Bt):
            for h in range(H):
                K, _ = wl.unit_kv(w, l, bb, h)
                q = wl.unit_decode_queries(w, l, bb, h, K, step + 1)[:, step]
                Q[l, bb, h * G:(h + 1) * G] = q[:G]
    return Q


def oracle_decode_all(lay, Q, cfg):
    L, Bt, Hq, d = Q.shape
    H = cfg.n_kv_heads
    G = Hq // H
    qf = bf16_to_f64(Q)
    out = np.zeros((L, Bt, Hq, d))
    oc = ocfg_from(cfg)
    for l in range(L):
        for bb in range(Bt):
            for h in range(H):
                u = (l * Bt + bb) * H + h
                uc = unit_from_layout(lay, u)
                out[l, bb, h * G:(h + 1) * G] = orc.decode_unit(uc, qf[l, bb, h * G:(h + 1) * G], oc)
    return out


def run_decode(cache, Q, layer=-1):
    Qd = Q.cuda().contiguous()
    O = torch.full(Qd.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(cache, layer, Qd, O)
    torch.cuda.synchronize()
    return O


def test_tiny_oracle_built_cache():
    """Tiny workload: s = 4096, b = 256 = 224 main + 32 residual (fixed), 16 decode queries."""
    w = wl.WORKLOADS["tiny"]
    K, V = wl.unit_kv(w, 0, 0, 0)
    Qo = wl.unit_obs_queries(w, 0, 0, 0, K)
    Qd = wl.unit_decode_queries(w, 0, 0, 0, K, w.steps)
    oc = orc.OracleConfig(budget=w.budget, residual_override=32)
    cache = orc.build_unit(bf16_to_f64(K), bf16_to_f64(V), bf16_to_f64(Qo), oc)
    assert cache.r == 32 and len(cache.main_pos) == 224
    lay = empty_layout(1, w.budget)
    put_unit(lay, 0, cache)
    cfg = mkcfg(batch=1, n_layers=1, n_kv_heads=1, group=4, seq_len=w.seq_len,
                                 budget=w.budget)
    h = R.reskv_import_cache(cfg, **lay)
    qf = bf16_to_f64(Qd)
    worst = (0.0, 0.0)
    for t in range(w.steps):
        q = Qd[:, t].reshape(1, 4, 128).contiguous()
        O = run_decode(h, q, layer=0).cpu().numpy()[0]
        ref = orc.decode_unit(cache, qf[:, t], oc)
        mx, rel = assert_output_parity(O, ref, f"step {t}")
        worst = (max(worst[0], mx), max(worst[1], rel))
    assert worst[1] < 1e-4          # fp32 accumulation lands far inside the bar
    R.reskv_check_status(h)
    h.free()


SPLITS = [(1, 0), (300, 0), (250, 50), (100, 7), (17, 1), (200, 60), (64, 12), (299, 1),
          (150, 150), (33, 0), (5, 200), (260, 40)]


@pytest.mark.parametrize("decode_warps", [0, 1, 3, 17, 64, 5000])
def test_ragged_layout_all_layers(decode_warps):
    """12 units (2 layers x 3 batch x 2 KV heads), b = 300 (rows straddle the
    8-slot stages), ragged main/residual splits with empty entries and unused
    tail slots; one all-layer launch cut into various warp counts."""
    L, Bt, H, G, b = 2, 3, 2, 4, 300
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b, decode_warps=decode_warps)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    O = run_decode(h, Q).cpu().numpy()
    ref = oracle_decode_all(lay, Q, cfg)
    assert not np.isnan(O).any()
    mx, rel = assert_output_parity(O, ref, f"warps {decode_warps}")
    assert rel < 1e-4
    R.reskv_check_status(h)


def test_per_layer_calls_match_all_layer_call():
    L, Bt, H, G, b = 2, 3, 2, 4, 300
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    O_all = run_decode(h, Q).cpu().numpy()
    for l in range(L):
        O_l = run_decode(h, Q[l].contiguous(), layer=l).cpu().numpy()
        mx, rel = errors(O_l, O_all[l].astype(np.float64))
        assert rel < SPLIT_REL


def test_layer_range_calls_match_all_layer_call():
    """reskv_decode_attn_layers over contiguous layer ranges (one launch each)
    gives the all-layer call's outputs; ranges outside the cache are refused."""
    L, Bt, H, G, b = 6, 3, 2, 4, 300
    rng = np.random.default_rng(31)
    splits = []
    for _ in range(L * Bt * H):
        n = int(rng.integers(1, b + 1))
        m = int(rng.integers(1, n + 1))
        splits.append((m, n - m))
    w, lay = synthetic_layout(L, Bt, H, b, splits)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len, budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    O_all = run_decode(h, Q).cpu().numpy()
    for l0, n in ((0, 6), (0, 2), (1, 3), (5, 1), (2, 4), (3, 2)):
        O = torch.full((n,) + tuple(Q.shape[1:]), float("nan"), dtype=torch.float32, device="cuda")
        R.reskv_decode_attn_layers(h, l0, n, Q[l0:l0 + n].cuda().contiguous(), O)
        torch.cuda.synchronize()
        assert errors(O.cpu().numpy(), O_all[l0:l0 + n].astype(np.float64))[1] < SPLIT_REL
    Qd = Q[:2].cuda().contiguous()
    Od = torch.empty(Qd.shape, dtype=torch.float32, device="cuda")
    for l0, n in ((-1, 2), (5, 2)):
        with pytest.raises(R.ReskvError) as e:
            R.reskv_decode_attn_layers(h, l0, n, Qd, Od)
        assert e.value.status == R.RESKV_ERR_INVALID_ARG
    import ctypes
    st = R.load_library().reskv_decode_attn_layers(h.handle, 0, 0, ctypes.c_void_p(Qd.data_ptr()),
                                                   ctypes.c_void_p(Od.data_ptr()), None)
    assert st == R.RESKV_ERR_INVALID_ARG
    R.reskv_check_status(h)


def test_kv_chunks_are_single_3d_copies():
    """On this part the driver takes the 3-D K/V maps: one TMA copy per
    16-row chunk of K or of V (the 2-D form, two copies each, is the
    fallback).  The decode results are those the other tests check."""
    L, Bt, H, G, b = 1, 1, 2, 4, 64
    w, lay = synthetic_layout(L, Bt, H, b, [(60, 4), (64, 0)])
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len, budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    assert R.reskv_get_info(h)["kv_copy_rank"] == 3


def test_host_buffer_call_matches_device_call():
    """reskv_decode_attn_host gives the device call's outputs bit for bit and
    matches the oracle, with page-locked buffers (the kernel reads Q and
    writes O in host memory) and with pageable ones (staged; repeated calls
    reuse the staging); overlapping host buffers are refused."""
    L, Bt, H, G, b = 5, 3, 2, 4, 300          # odd layer count: uneven groups
    rng = np.random.default_rng(37)
    splits = []
    for _ in range(L * Bt * H):
        n = int(rng.integers(1, b + 1))
        m = int(rng.integers(1, n + 1))
        splits.append((m, n - m))
    w, lay = synthetic_layout(L, Bt, H, b, splits)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len, budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    for step in (0, 1):
        Q = queries_for(w, L, Bt, H, G, step=step)
        O_dev = run_decode(h, Q).cpu().numpy().astype(np.float64)
        ref = oracle_decode_all(lay, Q, cfg)
        for pinned in (True, False):
            Qh = Q.contiguous()
            Oh = torch.full(Q.shape, float("nan"), dtype=torch.float32)
            if pinned:
                Qh, Oh = Qh.pin_memory(), Oh.pin_memory()
            R.reskv_decode_attn_host(h, Qh, Oh)
            torch.cuda.synchronize()
            O = Oh.numpy().astype(np.float64)
            assert not np.isnan(O).any()
            assert np.array_equal(O, O_dev), f"pinned {pinned}: differs from the device call"
            assert_output_parity(O, ref, f"host call, step {step}, pinned {pinned}")
    buf = torch.zeros(Q.numel() * 3, dtype=torch.bfloat16)
    Qv = buf[:Q.numel()]
    Ov = buf.view(torch.float32)[Q.numel() // 4:Q.numel() // 4 + Q.numel()]
    with pytest.raises(R.ReskvError) as e:
        R.reskv_decode_attn_host(h, Qv, Ov)
    assert e.value.status == R.RESKV_ERR_INVALID_ARG
    R.reskv_check_status(h)


def test_determinism_and_split_invariance():
    L, Bt, H, G, b = 2, 3, 2, 4, 300
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    Q = queries_for(w, L, Bt, H, G)
    outs = []
    for dw in (1, 2, 4, 16, 0):
        cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G,
                                     seq_len=w.seq_len, budget=b, decode_warps=dw)
        h = R.reskv_import_cache(cfg, **lay)
        o1 = run_decode(h, Q)
        o2 = run_decode(h, Q)
        assert torch.equal(o1, o2), "decode must be bitwise deterministic"
        outs.append(o1.cpu().numpy().astype(np.float64))
    for o in outs[1:]:
        assert errors(o, outs[0])[1] < SPLIT_REL


@pytest.mark.parametrize("G", [1, 2])
def test_group_sizes(G):
    L, Bt, H, b = 1, 2, 3, 256
    splits = [(200, 56), (256, 0), (10, 100), (128, 64), (1, 255), (100, 3)]
    w, lay = synthetic_layout(L, Bt, H, b, splits)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    O = run_decode(h, Q).cpu().numpy()
    assert_output_parity(O, oracle_decode_all(lay, Q, cfg), f"G={G}")


def _textbook(q, K, V):
    return softmax(K @ q / math.sqrt(K.shape[1])) @ V


def test_fixed_point_empty_residual_is_eviction():
    """Sec. 5.4: R empty gives eviction attention over M (Eq. evict)."""
    L, Bt, H, G, b = 1, 2, 2, 4, 512
    splits = [(512, 0), (300, 0), (77, 0), (1, 0)]
    w, lay = synthetic_layout(L, Bt, H, b, splits)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    O = run_decode(h, Q).cpu().numpy()
    qf = bf16_to_f64(Q)
    for u, (m, _) in enumerate(splits):
        bb, hh = divmod(u, H)
        Km = orc.bf16_bits_to_f64(lay["kslots"][u, :m])
        Vm = orc.bf16_bits_to_f64(lay["vslots"][u, :m])
        for g in range(G):
            ref = _textbook(qf[0, bb, hh * G + g], Km, Vm)
            assert_output_parity(O[0, bb, hh * G + g], ref, "eviction")


def test_fixed_point_gate_zero_is_main_only():
    L, Bt, H, G, b = 1, 1, 3, 4, 400
    splits = [(300, 100), (50, 350), (399, 1)]
    w, lay = synthetic_layout(L, Bt, H, b, splits)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b, gate_mode=R.RESKV_GATE_FIXED, g_fixed=0.0)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    O = run_decode(h, Q).cpu().numpy()
    qf = bf16_to_f64(Q)
    for u, (m, _) in enumerate(splits):
        Km = orc.bf16_bits_to_f64(lay["kslots"][u, :m])
        Vm = orc.bf16_bits_to_f64(lay["vslots"][u, :m])
        for g in range(G):
            assert_output_parity(O[0, 0, u * G + g], _textbook(qf[0, 0, u * G + g], Km, Vm), "g=0")


def test_fixed_point_exact_residual_encoding_is_full_attention():
    """Sec. 4.2, Eq. residual: one entry carrying log Z_E(q) and N_E/Z_E of the
    evicted tokens for the query of each head (G = 1) recovers o_S; the only
    error left is the bf16 storage of the entry's value."""
    s, m, d = 2048, 300, 128
    w = wl.scaled(wl.WORKLOADS["tiny"], seq_len=s)
    K, V = wl.unit_kv(w, 0, 0, 0)
    Qd = wl.unit_decode_queries(w, 0, 0, 0, K, 1)[0, 0]
    Kf, Vf, q = bf16_to_f64(K), bf16_to_f64(V), bf16_to_f64(Qd)
    a = Kf[m:] @ q / math.sqrt(d)
    ZE = np.exp(a).sum()
    NE = np.exp(a) @ Vf[m:]
    lay = empty_layout(1, m + 1)
    lay["n_main"][0], lay["n_res"][0] = m, 1
    lay["kslots"][0, :m] = bf16_bits(K[:m])
    lay["vslots"][0, :m] = bf16_bits(V[:m])
    vbar = orc.round_to_bf16(NE / ZE)
    lay["vslots"][0, m] = (vbar.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    lay["logc"][0, m] = np.float32(np.log(ZE))          # k_bar = 0, so <q, k_bar> = 0
    cfg = mkcfg(batch=1, n_layers=1, n_kv_heads=1, group=1, seq_len=s,
                                 budget=m + 1, gate_mode=R.RESKV_GATE_FIXED, g_fixed=1.0)
    h = R.reskv_import_cache(cfg, **lay)
    O = run_decode(h, Qd.reshape(1, 1, 1, d)).cpu().numpy()[0, 0, 0]
    full = _textbook(q, Kf, Vf)
    assert_output_parity(O, full, "exact encoding")
    # the residual's share of the output carries only bf16 rounding of v_bar
    assert errors(O, full)[1] < 4e-3 * ZE / (ZE + np.exp(Kf[:m] @ q / math.sqrt(d)).sum()) + 1e-5


@pytest.mark.parametrize("L,Bt,H", [(1, 1, 1), (1, 3, 4), (2, 4, 8), (1, 25, 4), (2, 20, 8)])
def test_launch_sizes(L, Bt, H):
    """Launches of 1 to 320 units with b = 200 (chunks straddle units): the
    automatic plan moves from clusters of 8 CTAs per unit through smaller ones
    to the stream-K split (and, for the cluster kernel chosen explicitly,
    single-CTA clusters in several waves); per-layer and all-layer calls."""
    G, b = 4, 200
    U = L * Bt * H
    rng = np.random.default_rng(U)
    splits = []
    for _ in range(U):
        n = int(rng.integers(1, b + 1))
        m = int(rng.integers(1, n + 1))
        splits.append((m, n - m))
    w, lay = synthetic_layout(L, Bt, H, b, splits)
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len, budget=b)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    ref = oracle_decode_all(lay, Q, cfg)
    O = run_decode(h, Q).cpu().numpy()
    assert_output_parity(O, ref, f"all layers, {U} units")
    for l in range(L):
        O_l = run_decode(h, Q[l].contiguous(), layer=l).cpu().numpy()
        assert_output_parity(O_l, ref[l], f"layer {l}, {Bt * H} units")
    R.reskv_check_status(h)


@pytest.mark.parametrize("gate", ["dynamic", "fixed_0.4", "fixed_1"])
def test_separate_softmax_ablation(gate):
    """The "w/o shared softmax" ablation (separately normalised branches mixed by
    the gate) on the ragged 12-unit layout, all-layer and per-layer calls."""
    L, Bt, H, G, b = 2, 3, 2, 4, 300
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    kw = {} if gate == "dynamic" else dict(gate_mode=R.RESKV_GATE_FIXED,
                                           g_fixed=float(gate.split("_")[1]))
    cfg = mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len, budget=b,
                softmax_mode=R.RESKV_SOFTMAX_SEPARATE, **kw)
    h = R.reskv_import_cache(cfg, **lay)
    Q = queries_for(w, L, Bt, H, G)
    ref = oracle_decode_all(lay, Q, cfg)
    O = run_decode(h, Q).cpu().numpy()
    assert_output_parity(O, ref, f"separate softmax, gate {gate}")
    for l in range(L):
        O_l = run_decode(h, Q[l].contiguous(), layer=l).cpu().numpy()
        assert_output_parity(O_l, ref[l], f"separate softmax, gate {gate}, layer {l}")
    # the ablation differs from the method where residual mass is present
    shared = oracle_decode_all(lay, Q, mkcfg(batch=Bt, n_layers=L, n_kv_heads=H, group=G,
                                             seq_len=w.seq_len, budget=b, **kw))
    assert errors(ref, shared)[1] > 1e-3
    R.reskv_check_status(h)
