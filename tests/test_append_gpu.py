"""Decode-time append (Sec. 3.1: each decode step appends the new token's key
and value) through the C ABI: rows added with reskv_append join the exact main
cache of their unit, and every decode path attends to them.  The reference is
the fp64 oracle's append_tokens on the same rows.  Past append_capacity the
appended slots are a ring of the latest tokens, and the oldest is dropped or
folded into its nearest residual entry (the oracle's append_ring): entries,
counts and rows must match the oracle bit for bit, and every decode path its
decode.
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
                                 budget=b, append_capacity=A, append_policy=R.RESKV_APPEND_FAIL)
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


POLICIES = {"drop": R.RESKV_APPEND_RING_DROP, "fold": R.RESKV_APPEND_RING_FOLD}
ORACLE_POLICY = {"drop": orc.APPEND_RING_DROP, "fold": orc.APPEND_RING_FOLD}


def check_ring_state(ex, units, n_app, lay):
    """The exported layout against the oracle's units: the same residual
    entries (bf16 bits), counts and log-counts, and the same appended tokens
    (the ring holds them in another order: compared by position)."""
    for u, ref in enumerate(units):
        m, r = int(lay["n_main"][u]), int(lay["n_res"][u])
        assert int(ex["n_app"][u]) == n_app[u]
        gk = ex["kslots"][u, m:m + r]
        gv = ex["vslots"][u, m:m + r]
        assert np.array_equal(orc.bf16_bits_to_f64(gk), ref.kbar), f"unit {u}: k_bar"
        assert np.array_equal(orc.bf16_bits_to_f64(gv), ref.vbar), f"unit {u}: v_bar"
        assert np.array_equal(ex["counts"][u, m:m + r], ref.counts), f"unit {u}: counts"
        want = np.where(ref.counts > 0, np.log(np.maximum(ref.counts, 1)), -np.inf)
        got = ex["logc"][u, m:m + r].astype(np.float64)
        fin = np.isfinite(want)
        assert np.array_equal(np.isfinite(got), fin)
        np.testing.assert_allclose(got[fin], want[fin], rtol=3e-7, atol=0)
        sl = slice(m + r, m + r + n_app[u])
        pos = ex["slot_pos"][u, sl]
        order = np.argsort(pos)
        assert np.array_equal(pos[order], ref.main_pos[m:]), f"unit {u}: appended positions"
        assert np.array_equal(orc.bf16_bits_to_f64(ex["kslots"][u, sl][order]), ref.kmain[m:])
        assert np.array_equal(orc.bf16_bits_to_f64(ex["vslots"][u, sl][order]), ref.vmain[m:])


@pytest.mark.parametrize("kernel", list(KERNELS))
@pytest.mark.parametrize("policy", list(POLICIES))
def test_ring_appends_run_past_the_capacity(kernel, policy):
    """3 A tokens appended into A = 8 slots per unit (per layer and all layers
    at once): no call is refused; decodes along the way match the oracle's
    decode of its grown units, and the state matches bit for bit."""
    L, Bt, H, G, b, A = 2, 3, 2, 4, 300, 8
    w, lay = synthetic_layout(L, Bt, H, b, SPLITS)
    lay = with_capacity(lay, A)
    cfg = R.reskv_config_default(batch=Bt, n_layers=L, n_kv_heads=H, group=G, seq_len=w.seq_len,
                                 budget=b, append_capacity=A, append_policy=POLICIES[policy],
                                 decode_kernel=KERNELS[kernel])
    h = R.reskv_import_cache(cfg, **lay)
    U = L * Bt * H
    units = [unit_from_layout(lay, u) for u in range(U)]
    n_app = [0] * U
    ocfg = orc.OracleConfig(budget=b)
    g = torch.Generator().manual_seed(11)
    for step in range(3 * A):
        Kn = torch.randn((L, Bt, H, 128), generator=g).to(torch.bfloat16)
        Vn = (2.0 * torch.randn((L, Bt, H, 128), generator=g)).to(torch.bfloat16)
        if step % 3 == 0:
            R.reskv_append(h, -1, Kn.cuda(), Vn.cuda())
        else:
            for l in range(L):
                R.reskv_append(h, l, Kn[l].cuda(), Vn[l].cuda())
        kf, vf = bf16_to_f64(Kn), bf16_to_f64(Vn)
        for l in range(L):
            for bb in range(Bt):
                for hh in range(H):
                    u = (l * Bt + bb) * H + hh
                    units[u], n_app[u] = orc.append_ring(
                        units[u], kf[l, bb, hh][None], vf[l, bb, hh][None],
                        np.array([w.seq_len + step]), n_app[u], A, ORACLE_POLICY[policy])
        if step % 4 == 3 or step == 3 * A - 1:
            Q = torch.randn((L, Bt, H * G, 128), generator=g)
            Q[:, :, ::2] = 2.0 * Kn.float().repeat_interleave(G, dim=2)[:, :, ::2] + 0.3 * Q[:, :, ::2]
            Q = Q.to(torch.bfloat16)
            ref = oracle_outputs(units, Q, L, Bt, H, G, ocfg)
            assert_output_parity(decode(h, Q), ref, f"{kernel} {policy}, step {step}")
            for l in range(L):
                assert_output_parity(decode(h, Q[l], l), ref[l], f"{kernel} {policy} {step} {l}")
    R.reskv_check_status(h)
    assert R.reskv_get_info(h)["max_appended"] == A
    check_ring_state(R.reskv_export_cache(h), units, n_app, lay)
    if policy == "fold":                  # every token stays in the cache
        ex = R.reskv_export_cache(h)
        for u in range(U):
            m, r = int(lay["n_main"][u]), int(lay["n_res"][u])
            if r:
                assert ex["counts"][u, m:m + r].sum() == lay["counts"][u, m:m + r].sum() + 2 * A
    h.free()


def _crafted_unit(entries, b=16, A=1):
    """One unit: 8 main rows of ones, residual entries `entries` (rows of exact
    bf16 values, count 1), room for A appended tokens."""
    r = len(entries)
    lay = {k: v for k, v in with_capacity(
        dict(n_main=np.array([8], np.int32), n_res=np.array([r], np.int32),
             kslots=np.zeros((1, b, 128), np.uint16), vslots=np.zeros((1, b, 128), np.uint16),
             logc=np.zeros((1, b), np.float32), slot_pos=np.full((1, b), -1, np.int32),
             counts=np.zeros((1, b), np.int32)), A).items()}
    ones = torch.ones((8, 128), dtype=torch.bfloat16)
    lay["kslots"][0, :8] = bf16_bits(ones)
    lay["vslots"][0, :8] = bf16_bits(ones)
    lay["slot_pos"][0, :8] = np.arange(8)
    E = torch.from_numpy(np.asarray(entries, np.float32)).to(torch.bfloat16)
    assert np.array_equal(E.double().numpy(), np.asarray(entries))          # exact in bf16
    lay["kslots"][0, 8:8 + r] = bf16_bits(E)
    lay["vslots"][0, 8:8 + r] = bf16_bits(E)
    lay["counts"][0, 8:8 + r] = 1
    return lay


@pytest.mark.parametrize("case", ["fp64_near_tie", "exact_tie", "wide_span", "subnormal"])
def test_fold_picks_the_exactly_nearest_entry(case):
    """Crafted entries where the nearest one is decided below float64
    resolution, by a tie (lower entry), across an exponent span wider than
    the 128-bit window (the wide accumulator), and among bf16 subnormals."""
    d = 128
    e = np.zeros((3, d))
    k = np.zeros(d)
    if case == "fp64_near_tie":        # 2^54 + 1 vs 2^54 + 1/4
        e[:2, 0] = 2.0 ** 27
        e[0, 1], e[1, 1] = 1.0, 0.5
        e[2, 0] = 2.0 ** 28
    elif case == "exact_tie":
        e[0, 3], e[1, 3], e[2, 3] = 1.0, -1.0, 1.0
    elif case == "wide_span":          # 2^-120 vs 2^-122, next to a value 2^30
        k[0] = 1.0
        e[:2, 0] = 1.0
        e[0, 1], e[1, 2] = 2.0 ** -60, 2.0 ** -61
        e[2, 0] = 2.0 ** 30
    else:
        e[0, 0], e[1, 0], e[2, 0] = 3 * 2.0 ** -133, 2.0 ** -133, 2.0 ** -131
    want = orc.nearest_entry(k, e)
    lay = _crafted_unit(e)
    cfg = R.reskv_config_default(batch=1, n_layers=1, n_kv_heads=1, group=4, seq_len=64, budget=16,
                                 append_capacity=1, append_policy=R.RESKV_APPEND_RING_FOLD)
    h = R.reskv_import_cache(cfg, **lay)
    kt = torch.from_numpy(k.astype(np.float32)).to(torch.bfloat16).reshape(1, 1, 128).cuda()
    R.reskv_append(h, 0, kt, kt)                # the token to be folded
    R.reskv_append(h, 0, kt * 0, kt * 0)        # pushes it out of the ring
    torch.cuda.synchronize()
    R.reskv_check_status(h)
    ex = R.reskv_export_cache(h)
    counts = ex["counts"][0, 8:11]
    assert counts.tolist() == [2 if j == want else 1 for j in range(3)], (case, want, counts)
    ref = orc.fold_into_entry(e[want], e[want], 1, k, k, 1.0)
    assert np.array_equal(orc.bf16_bits_to_f64(ex["kslots"][0, 8 + want]), ref[0])
    h.free()
