"""Split plans of the tensor-core stream-K decode kernel through the C ABI.

Many short units (one all-layer launch of 16384 units of 32 slots): the
automatic plan gives every warp k whole consecutive units, so that no unit is
cut between warps.  Its outputs must match the fp64 oracle on sampled units
and the equal-slot-piece split (units cut between warps, merged through
partial records) on every unit; uniform and per-unit budgets.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2607_29591_gb300 import build as B
from paper_2607_29591_gb300 import reskv as R

from helpers import assert_output_parity, bf16_to_f64, errors, unit_from_layout

pytestmark = pytest.mark.gpu

L, BT, H, G, D = 4, 64, 64, 4, 128


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    return R.load_library()


def random_layout(budgets, seed):
    """Flat layout of units with the given budgets: seeded normal rows, random
    main / residual splits (every unit full or not), counts with some zeros."""
    U = len(budgets)
    off = np.concatenate([[0], np.cumsum(budgets.astype(np.int64))])
    N = int(off[-1])
    g = torch.Generator().manual_seed(seed)
    bits = lambda t: t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    rng = np.random.default_rng(seed)
    n = np.where(rng.random(U) < 0.7, budgets, rng.integers(1, budgets + 1))
    m = rng.integers(1, n + 1).astype(np.int32)
    r = (n - m).astype(np.int32)
    counts = np.zeros(N, np.int32)
    logc = np.zeros(N, np.float32)
    c = rng.integers(0, 100, N)
    c[rng.random(N) < 0.05] = 0
    for u in np.nonzero(r)[0]:
        o = int(off[u]) + int(m[u])
        counts[o:o + r[u]] = c[o:o + r[u]]
    res = counts > 0
    logc[res] = np.log(counts[res]).astype(np.float32)
    is_res = np.zeros(N, bool)
    for u in np.nonzero(r)[0]:
        o = int(off[u]) + int(m[u])
        is_res[o:o + r[u]] = True
    logc[is_res & ~res] = -np.inf
    return dict(n_main=m, n_res=r, kslots=bits(torch.randn((N, D), generator=g)),
                vslots=bits(torch.randn((N, D), generator=g)), logc=logc,
                slot_pos=np.full(N, -1, np.int32), counts=counts, offsets=off)


def decode(cache, Q):
    O = torch.full(Q.shape, float("nan"), dtype=torch.float32, device="cuda")
    R.reskv_decode_attn(cache, -1, Q, O)
    torch.cuda.synchronize()
    R.reskv_check_status(cache)
    return O.cpu().numpy()


@pytest.mark.parametrize("ragged", [False, True], ids=["uniform", "per_unit_budgets"])
def test_whole_units_per_warp(ragged):
    U = L * BT * H
    rng = np.random.default_rng(7)
    budgets = (rng.integers(16, 49, U) if ragged else np.full(U, 32)).astype(np.int32)
    lay = random_layout(budgets, 11 + int(ragged))
    arrs = {k: lay[k] for k in ("n_main", "n_res", "kslots", "vslots", "logc", "slot_pos",
                                "counts")}
    shape = dict(batch=BT, n_layers=L, n_kv_heads=H, group=G, seq_len=4096,
                 budget=int(budgets.max()), unit_budgets=budgets if ragged else None)
    if not ragged:
        arrs = {k: (v.reshape(U, 32, D) if k in ("kslots", "vslots") else
                    v.reshape(U, 32) if k in ("logc", "slot_pos", "counts") else v)
                for k, v in arrs.items()}
    auto = R.reskv_import_cache(R.reskv_config_default(**shape), **arrs)
    info = R.reskv_get_info(auto)
    assert info["all_cluster"] == 0 and info["all_units_per_warp"] > 1, info
    pieces = R.reskv_import_cache(R.reskv_config_default(decode_kernel=R.RESKV_DECODE_MMA,
                                                         decode_warps=1216, **shape), **arrs)
    assert R.reskv_get_info(pieces)["all_units_per_warp"] == 0
    g = torch.Generator().manual_seed(3)
    Q = torch.randn((L, BT, H * G, D), generator=g).to(torch.bfloat16).cuda()
    Oa, Op = decode(auto, Q), decode(pieces, Q)
    assert not np.isnan(Oa).any()
    assert errors(Oa, Op.astype(np.float64))[1] < 1e-5
    # sampled units against the oracle (the layout as the oracle sees it)
    qf = bf16_to_f64(Q)
    oc = orc.OracleConfig(budget=int(budgets.max()))
    for u in rng.choice(U, 48, replace=False):
        l, rem = divmod(int(u), BT * H)
        b, h = divmod(rem, H)
        ref = orc.decode_unit(unit_from_layout(lay, int(u)), qf[l, b, h * G:(h + 1) * G], oc)
        assert_output_parity(Oa[l, b, h * G:(h + 1) * G], ref, f"unit {u}")
    auto.free()
    pieces.free()


def test_whole_units_per_warp_with_appended_rows():
    """The whole-unit split on units that also hold rows appended at decode
    time (append capacity 4, two appends): against the equal-piece split."""
    U = L * BT * H
    budgets = np.full(U, 32, np.int32)
    lay = random_layout(budgets, 21)
    A = 4
    S = 32 + A
    arrs = {}
    for k in ("kslots", "vslots"):
        a = lay[k].reshape(U, 32, D)
        arrs[k] = np.concatenate([a, np.zeros((U, A, D), np.uint16)], axis=1)
    for k, fill in (("logc", 0), ("slot_pos", -1), ("counts", 0)):
        a = lay[k].reshape(U, 32)
        arrs[k] = np.concatenate([a, np.full((U, A), fill, a.dtype)], axis=1)
    arrs["n_main"], arrs["n_res"] = lay["n_main"], lay["n_res"]
    shape = dict(batch=BT, n_layers=L, n_kv_heads=H, group=G, seq_len=4096, budget=32,
                 append_capacity=A)
    auto = R.reskv_import_cache(R.reskv_config_default(**shape), **arrs)
    assert R.reskv_get_info(auto)["all_units_per_warp"] > 1
    pieces = R.reskv_import_cache(R.reskv_config_default(decode_kernel=R.RESKV_DECODE_MMA,
                                                         decode_warps=1216, **shape), **arrs)
    g = torch.Generator().manual_seed(9)
    for _ in range(2):
        kn = torch.randn((L, BT, H, D), generator=g).to(torch.bfloat16).cuda()
        vn = torch.randn((L, BT, H, D), generator=g).to(torch.bfloat16).cuda()
        R.reskv_append(auto, -1, kn, vn)
        R.reskv_append(pieces, -1, kn, vn)
    Q = torch.randn((L, BT, H * G, D), generator=g).to(torch.bfloat16).cuda()
    Oa, Op = decode(auto, Q), decode(pieces, Q)
    assert not np.isnan(Oa).any()
    assert errors(Oa, Op.astype(np.float64))[1] < 1e-5
    auto.free()
    pieces.free()
