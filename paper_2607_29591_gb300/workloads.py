"""Seeded synthetic inputs shaped like the paper's long-context decode workloads.

This module holds no part of the method: it only draws keys, values and
queries.  It is device-agnostic torch code whose arithmetic is integer hashing
plus single float32 multiplies/adds, so the same call produces bit-identical
tensors on the CPU and on the GPU.  Tests feed its output both to the CUDA
library and to the fp64 oracle; neither of those imports the other.

Recipe (seed base 42, the paper's fixed seed, App. B):

* counter-based uniforms: ``u(key, i) = lowbias32(key ^ lowbias32(i))`` where
  ``lowbias32`` is C. Wellons' published 32-bit integer hash ("hash-prospector":
  xorshift 16, multiply 0x7feb352d, xorshift 15, multiply 0x846ca68b,
  xorshift 16); ``key`` chains the hash over (seed, tensor tag, layer, batch,
  head);
* approximately normal values: the Irwin-Hall sum of four 16-bit uniforms
  (two hashes), centred and scaled to unit variance in float32;
* keys and values: N(0,1) with 4 outlier channels per (layer, KV head) scaled
  by 8 (channels ``c, c+32, c+64, c+96`` with ``c`` drawn from the hash);
* queries (observation and decode): ``0.7 * k_{p*} + 0.3 * n`` with ``p*`` a
  uniformly drawn cached position, so attention is peaked as in retrieval;
* long-context stress: every non-needle key adds a slowly drifting mean
  ``cos(2 pi p/65536) a + sin(2 pi p/65536) b`` (a, b ~ N(0,1)^d per unit);
  1% of the positions outside the recent window are needles with keys
  ``3 n``; half of the queries pick a needle as their target;
* small-budget workload: per-(layer, KV head) residual counts drawn uniformly
  from 0..64, shared across the batch, with a seeded 1/8 of them forced to 0.

All tensors are rounded to bf16 (round to nearest even) as the last step.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch

SEED = 42

# tensor tags for the key chain
TAG_K, TAG_V, TAG_QOBS, TAG_QDEC = 1, 2, 3, 4
TAG_OUTLIER_K, TAG_OUTLIER_V = 5, 6
TAG_DRIFT_A, TAG_DRIFT_B = 7, 8
TAG_NEEDLE, TAG_NEEDLE_K = 9, 10
TAG_PICK_OBS, TAG_PICK_DEC = 11, 12
TAG_R, TAG_R_ZERO = 13, 14

_C1 = 0x7FEB352D
_C2 = 0x846CA68B
_C2_SIGNED = _C2 - (1 << 32)          # the same bit pattern as an int32 value

# Irwin-Hall of four uniforms on {0..65535}: mean 131070, variance 4*(65536^2-1)/12
_IH_MEAN = 131070
NORM_SCALE = float(np.float32(1.0 / math.sqrt(4.0 * (65536.0 ** 2 - 1.0) / 12.0)))
Q_KEY_W = float(np.float32(0.7))
Q_NOISE_W = float(np.float32(0.3))
OUTLIER_SCALE = 8.0
NEEDLE_SCALE = 3.0
DRIFT_PERIOD = 65536


# ---------------------------------------------------------------------------
# hashing
# ---------------------------------------------------------------------------

def lowbias32_int(x: int) -> int:
    """lowbias32 on a Python int (host-side key derivation)."""
    x &= 0xFFFFFFFF
    x ^= x >> 16
    x = (x * _C1) & 0xFFFFFFFF
    x ^= x >> 15
    x = (x * _C2) & 0xFFFFFFFF
    x ^= x >> 16
    return x


def key_of(*fields: int) -> int:
    """Chain the hash over (seed, tag, indices...)."""
    h = lowbias32_int(SEED)
    for f in fields:
        h = lowbias32_int(h ^ (int(f) & 0xFFFFFFFF))
    return h


def _to_i32(x: int) -> int:
    x &= 0xFFFFFFFF
    return x - (1 << 32) if x >= (1 << 31) else x


def lowbias32(x: torch.Tensor) -> torch.Tensor:
    """lowbias32 on an int32 tensor holding uint32 bit patterns (wrapping multiply)."""
    x = x ^ ((x >> 16) & 0xFFFF)
    x = x * _C1
    x = x ^ ((x >> 15) & 0x1FFFF)
    x = x * _C2_SIGNED
    x = x ^ ((x >> 16) & 0xFFFF)
    return x


def counter_hash(n: int, device) -> torch.Tensor:
    """lowbias32(i) for i in [0, n): the per-index half of u(key, i)."""
    return lowbias32(torch.arange(n, dtype=torch.int64, device=device).to(torch.int32))


def normals(keys: torch.Tensor, hidx: torch.Tensor) -> torch.Tensor:
    """Approximately N(0,1) float32 values.

    ``keys``: int32 [U] stream keys; ``hidx``: int32 [2n] = counter_hash(2n).
    Returns [U, n]; element i of stream k uses u(k, 2i) and u(k, 2i+1).
    """
    k = keys.reshape(-1, 1)
    u0 = lowbias32(k ^ hidx[0::2].reshape(1, -1))
    u1 = lowbias32(k ^ hidx[1::2].reshape(1, -1))
    s = (u0 & 0xFFFF) + ((u0 >> 16) & 0xFFFF) + (u1 & 0xFFFF) + ((u1 >> 16) & 0xFFFF)
    s = s - _IH_MEAN
    return s.to(torch.float32) * NORM_SCALE


def uniforms_u32(keys: torch.Tensor, hidx: torch.Tensor) -> torch.Tensor:
    """u(key, i) as int64 values in [0, 2^32): [U, n] for hidx = counter_hash(n)."""
    u = lowbias32(keys.reshape(-1, 1) ^ hidx.reshape(1, -1))
    return u.to(torch.int64) & 0xFFFFFFFF


def keys_tensor(fields_list, device) -> torch.Tensor:
    return torch.tensor([_to_i32(key_of(*f)) for f in fields_list], dtype=torch.int32,
                        device=device)


# ---------------------------------------------------------------------------
# workloads
# ---------------------------------------------------------------------------

@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    batch: int
    n_kv_heads: int
    group: int
    head_dim: int
    seq_len: int
    budget: int
    n_obs: int
    n_fit: int
    n_val: int
    score_mode: int            # 0 = observation-window scores, 1 = key norm
    residual: str              # "proxy", "fixed:<r>" or "drawn"
    steps: int
    kind: str = "plain"        # "plain" or "drift_needles"
    recent_window: int = 64

    @property
    def n_q_heads(self) -> int:
        return self.n_kv_heads * self.group

    @property
    def n_units(self) -> int:
        return self.n_layers * self.batch * self.n_kv_heads

    def unit_index(self, layer: int, b: int, h: int) -> int:
        """Unit order of the cache layout: u = (layer * B + b) * H_kv + h."""
        return (layer * self.batch + b) * self.n_kv_heads + h

    def residual_override(self) -> Optional[np.ndarray]:
        """Per-unit residual counts for fixed / drawn workloads, else None."""
        if self.residual == "proxy":
            return None
        out = np.zeros(self.n_units, dtype=np.int32)
        for l in range(self.n_layers):
            for h in range(self.n_kv_heads):
                if self.residual.startswith("fixed:"):
                    r = int(self.residual.split(":")[1])
                else:
                    r = lowbias32_int(key_of(TAG_R, l, h)) % 65
                    if lowbias32_int(key_of(TAG_R_ZERO, l, h)) % 8 == 0:
                        r = 0
                for b in range(self.batch):
                    out[self.unit_index(l, b, h)] = r
        return out


WORKLOADS = {
    "tiny": Workload("tiny", 1, 1, 1, 4, 128, 4096, 256, 128, 96, 32, 0, "fixed:32", 16),
    "llama8b_layer_32k": Workload("llama8b_layer_32k", 1, 1, 8, 4, 128, 32768, 512,
                                  128, 96, 32, 0, "proxy", 256),
    "llama8b_32l_32k_b8": Workload("llama8b_32l_32k_b8", 32, 8, 8, 4, 128, 32768, 1024,
                                   32, 24, 8, 0, "proxy", 256),
    "long_128k_b4": Workload("long_128k_b4", 32, 4, 8, 4, 128, 131072, 2048,
                             128, 96, 32, 0, "proxy", 256, kind="drift_needles"),
    "small_budget_b64": Workload("small_budget_b64", 32, 64, 8, 4, 128, 16384, 128,
                                 0, 0, 0, 1, "drawn", 256),
}


def scaled(w: Workload, **changes) -> Workload:
    """A copy of a workload with some sizes changed (smaller parity cases)."""
    d = dict(w.__dict__)
    d.update(changes)
    return Workload(**d)


# ---------------------------------------------------------------------------
# generation
# ---------------------------------------------------------------------------

def _outlier_channels(tag: int, layer: int, h: int, d: int) -> list:
    c = lowbias32_int(key_of(tag, layer, h)) % (d // 4)
    return [c + j * (d // 4) for j in range(4)]


def _channel_scale(tag: int, layer: int, h: int, d: int, device) -> torch.Tensor:
    sc = torch.ones(d, dtype=torch.float32, device=device)
    sc[_outlier_channels(tag, layer, h, d)] = OUTLIER_SCALE
    return sc


def _drift_tables(s: int, device):
    p = np.arange(s, dtype=np.float64)
    ang = 2.0 * np.pi * p / DRIFT_PERIOD
    cos_t = torch.from_numpy(np.cos(ang).astype(np.float32)).to(device)
    sin_t = torch.from_numpy(np.sin(ang).astype(np.float32)).to(device)
    return cos_t, sin_t


def needle_positions(w: Workload, layer: int, b: int, h: int, device) -> torch.Tensor:
    """Sorted needle positions of one unit (long-context stress workload)."""
    s = w.seq_len
    hh = counter_hash(s, device)
    u = uniforms_u32(keys_tensor([(TAG_NEEDLE, layer, b, h)], device), hh)[0]
    mask = (u % 100) == 0
    mask[s - w.recent_window:] = False
    return torch.nonzero(mask).flatten()


def unit_kv(w: Workload, layer: int, b: int, h: int, device="cpu", hidx=None):
    """Keys and values of one (layer, batch, KV head) unit: bf16 [s, d] each."""
    s, d = w.seq_len, w.head_dim
    if hidx is None:
        hidx = counter_hash(2 * s * d, device)
    keys = keys_tensor([(TAG_K, layer, b, h), (TAG_V, layer, b, h)], device)
    n = normals(keys, hidx).reshape(2, s, d)
    kf = n[0] * _channel_scale(TAG_OUTLIER_K, layer, h, d, device)
    vf = n[1] * _channel_scale(TAG_OUTLIER_V, layer, h, d, device)
    if w.kind == "drift_needles":
        hd = counter_hash(2 * d, device)
        ab = normals(keys_tensor([(TAG_DRIFT_A, layer, b, h), (TAG_DRIFT_B, layer, b, h)],
                                 device), hd)
        cos_t, sin_t = _drift_tables(s, device)
        mu = cos_t.reshape(s, 1) * ab[0].reshape(1, d)
        mu = mu + sin_t.reshape(s, 1) * ab[1].reshape(1, d)
        kf = mu + kf
        needles = needle_positions(w, layer, b, h, device)
        if needles.numel():
            nk = normals(keys_tensor([(TAG_NEEDLE_K, layer, b, h)], device),
                         hidx[: 2 * needles.numel() * d]).reshape(-1, d)
            kf[needles] = nk * NEEDLE_SCALE
    return kf.to(torch.bfloat16), vf.to(torch.bfloat16)


def _queries(w: Workload, layer: int, b: int, h: int, K: torch.Tensor, n_q: int,
             tag_noise: int, tag_pick: int, device) -> torch.Tensor:
    """[G, n_q, d] queries 0.7 k_{p*} + 0.3 n for the G query heads of KV head h."""
    G, d, s = w.group, w.head_dim, w.seq_len
    hq = [h * G + g for g in range(G)]
    hidx = counter_hash(2 * n_q * d, device)
    noise = normals(keys_tensor([(tag_noise, layer, b, q) for q in hq], device), hidx)
    noise = noise.reshape(G, n_q, d)
    picks = uniforms_u32(keys_tensor([(tag_pick, layer, b, q) for q in hq], device),
                         counter_hash(2 * n_q, device)).reshape(G, n_q, 2)
    pos = picks[..., 1] % s
    if w.kind == "drift_needles":
        needles = needle_positions(w, layer, b, h, device)
        if needles.numel():
            use = (picks[..., 0] & 1) == 1
            npos = needles[picks[..., 1] % needles.numel()]
            pos = torch.where(use, npos, pos)
    kp = K[pos.reshape(-1)].to(torch.float32).reshape(G, n_q, d)
    q = kp * Q_KEY_W
    q = q + noise * Q_NOISE_W
    return q.to(torch.bfloat16)


def unit_obs_queries(w: Workload, layer: int, b: int, h: int, K: torch.Tensor, device="cpu"):
    """Observation queries of one unit: bf16 [G, n_obs, d] (fit rows first)."""
    return _queries(w, layer, b, h, K, w.n_obs, TAG_QOBS, TAG_PICK_OBS, device)


def unit_decode_queries(w: Workload, layer: int, b: int, h: int, K: torch.Tensor,
                        n_steps: int, device="cpu"):
    """Decode queries of one unit for steps 0..n_steps-1: bf16 [G, n_steps, d]."""
    return _queries(w, layer, b, h, K, n_steps, TAG_QDEC, TAG_PICK_DEC, device)


def layer_inputs(w: Workload, layer: int, device, n_dec_steps: int = 0):
    """All units of one layer.

    Returns K, V bf16 [B, H_kv, s, d]; Qobs bf16 [B, H_q, n_obs, d] (or None);
    Qdec bf16 [n_dec_steps, B, H_q, d] (or None).
    """
    B, H, G, s, d = w.batch, w.n_kv_heads, w.group, w.seq_len, w.head_dim
    K = torch.empty((B, H, s, d), dtype=torch.bfloat16, device=device)
    V = torch.empty_like(K)
    Qobs = torch.empty((B, H * G, w.n_obs, d), dtype=torch.bfloat16, device=device) \
        if w.n_obs > 0 else None
    Qdec = torch.empty((n_dec_steps, B, H * G, d), dtype=torch.bfloat16, device=device) \
        if n_dec_steps > 0 else None
    hidx = counter_hash(2 * s * d, device)
    for b in range(B):
        for h in range(H):
            k, v = unit_kv(w, layer, b, h, device, hidx)
            K[b, h], V[b, h] = k, v
            if Qobs is not None:
                Qobs[b, h * G:(h + 1) * G] = unit_obs_queries(w, layer, b, h, k, device)
            if Qdec is not None:
                qd = unit_decode_queries(w, layer, b, h, k, n_dec_steps, device)
                Qdec[:, b, h * G:(h + 1) * G] = qd.permute(1, 0, 2)
    return K, V, Qobs, Qdec
