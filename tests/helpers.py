"""Shared test utilities: bf16 conversions, layout assembly, tolerances."""
import math

import numpy as np
import torch

import oracle as orc

# Output tolerance against the fp64 oracle (max abs, relative L2).
MAX_ABS = 1e-2
REL_L2 = 2e-3


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().float().double().numpy()


def f64_to_bf16_bits(x) -> np.ndarray:
    """Bit patterns of values that are already exact bf16 numbers."""
    x32 = np.asarray(x, dtype=np.float32)
    assert np.array_equal(x32.astype(np.float64), np.asarray(x, dtype=np.float64))
    bits = x32.view(np.uint32)
    assert np.all((bits & 0xFFFF) == 0), "not a bf16 value"
    return (bits >> 16).astype(np.uint16)


def empty_layout(U: int, b: int, d: int = 128) -> dict:
    """Import layout of U units with unit stride b (budget + append capacity)."""
    return dict(n_main=np.zeros(U, np.int32), n_res=np.zeros(U, np.int32),
                kslots=np.zeros((U, b, d), np.uint16), vslots=np.zeros((U, b, d), np.uint16),
                logc=np.zeros((U, b), np.float32), slot_pos=np.full((U, b), -1, np.int32),
                counts=np.zeros((U, b), np.int32))


def put_unit(layout: dict, u: int, cache: "orc.UnitCache"):
    """Write an oracle-built unit into the import layout."""
    m, r = len(cache.main_pos), cache.r
    layout["n_main"][u], layout["n_res"][u] = m, r
    layout["kslots"][u, :m] = f64_to_bf16_bits(cache.kmain)
    layout["vslots"][u, :m] = f64_to_bf16_bits(cache.vmain)
    layout["slot_pos"][u, :m] = cache.main_pos
    if r:
        layout["kslots"][u, m:m + r] = f64_to_bf16_bits(cache.kbar)
        layout["vslots"][u, m:m + r] = f64_to_bf16_bits(cache.vbar)
        layout["logc"][u, m:m + r] = cache.logc.astype(np.float32)
        layout["counts"][u, m:m + r] = cache.counts


def unit_from_layout(layout: dict, u: int) -> "orc.UnitCache":
    """The oracle's view of one unit of a (host) layout: main rows, residual
    entries, then the rows appended at decode time (joined to the main cache)."""
    m, r = int(layout["n_main"][u]), int(layout["n_res"][u])
    a = int(layout["n_app"][u]) if layout.get("n_app") is not None else 0
    if "offsets" in layout:                      # per-unit budgets: flat arrays
        o0, o1 = int(layout["offsets"][u]), int(layout["offsets"][u + 1])
        view = {k: layout[k][o0:o1] for k in ("kslots", "vslots", "logc", "slot_pos", "counts")}
    else:
        view = {k: layout[k][u] for k in ("kslots", "vslots", "logc", "slot_pos", "counts")}
    k = orc.bf16_bits_to_f64(view["kslots"])
    v = orc.bf16_bits_to_f64(view["vslots"])
    unit = orc.UnitCache(main_pos=view["slot_pos"][:m].copy(), kmain=k[:m], vmain=v[:m],
                         kbar=k[m:m + r], vbar=v[m:m + r], counts=view["counts"][m:m + r],
                         logc=view["logc"][m:m + r].astype(np.float64), r=r)
    if a:
        unit = orc.append_tokens(unit, k[m + r:m + r + a], v[m + r:m + r + a],
                                 view["slot_pos"][m + r:m + r + a].copy())
    return unit


def errors(out: np.ndarray, ref: np.ndarray):
    diff = np.asarray(out, np.float64) - ref
    return float(np.max(np.abs(diff))), float(np.linalg.norm(diff) / np.linalg.norm(ref))


def assert_output_parity(out, ref, what=""):
    mx, rel = errors(out, ref)
    assert mx <= MAX_ABS and rel <= REL_L2, f"{what}: max abs {mx:.3g}, rel L2 {rel:.3g}"
    return mx, rel
