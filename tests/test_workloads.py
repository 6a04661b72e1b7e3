"""The seeded input generator: hash definition, determinism, distributions."""
import numpy as np
import torch

from paper_2607_29591_gb300 import workloads as wl


def _lowbias32_np(x):
    """lowbias32 written with numpy uint32 arithmetic (wraps mod 2^32)."""
    x = x.astype(np.uint32)
    x ^= x >> np.uint32(16)
    x *= np.uint32(0x7FEB352D)
    x ^= x >> np.uint32(15)
    x *= np.uint32(0x846CA68B)
    x ^= x >> np.uint32(16)
    return x


def test_hash_matches_uint32_reference():
    rng = np.random.default_rng(0)
    xs = rng.integers(0, 1 << 32, 100000, dtype=np.uint64).astype(np.uint32)
    got = wl.lowbias32(torch.from_numpy(xs.view(np.int32).copy()))
    assert np.array_equal(got.numpy().view(np.uint32), _lowbias32_np(xs))
    for x in (0, 1, 42, 0xFFFFFFFF, 0x80000000):
        assert wl.lowbias32_int(x) == int(_lowbias32_np(np.array([x], dtype=np.uint32))[0])


def test_normals_moments_and_determinism():
    keys = wl.keys_tensor([(1, 2, 3), (4, 5, 6)], "cpu")
    h = wl.counter_hash(2 * 200000, "cpu")
    a = wl.normals(keys, h)
    b = wl.normals(keys, h)
    assert torch.equal(a, b)
    x = a.double()
    assert abs(x.mean().item()) < 0.01
    assert abs(x.std().item() - 1.0) < 0.01
    assert x.abs().max().item() <= 2 * np.sqrt(3) + 1e-3        # Irwin-Hall support
    assert not torch.equal(a[0], a[1])


def test_unit_kv_outliers_and_dtype():
    w = wl.scaled(wl.WORKLOADS["tiny"], seq_len=2048)
    K, V = wl.unit_kv(w, 0, 0, 0)
    assert K.dtype == torch.bfloat16 and K.shape == (2048, 128)
    std = K.float().std(dim=0)
    ch = wl._outlier_channels(wl.TAG_OUTLIER_K, 0, 0, 128)
    assert len(set(ch)) == 4
    assert torch.all(std[ch] > 6.0) and torch.all(std[[c for c in range(128) if c not in ch]] < 1.3)
    K2, _ = wl.unit_kv(w, 0, 0, 0)
    assert torch.equal(K, K2)


def test_queries_are_peaked_on_their_target():
    w = wl.scaled(wl.WORKLOADS["tiny"], seq_len=1024)
    K, _ = wl.unit_kv(w, 0, 0, 0)
    Q = wl.unit_obs_queries(w, 0, 0, 0, K)
    assert Q.shape == (4, 128, 128)
    logits = Q.float().reshape(-1, 128) @ K.float().T / np.sqrt(128)
    w_max = torch.softmax(logits, dim=1).max(dim=1).values
    # peaked far above uniform (1/1024), with queries on both sides of the
    # gate threshold tau = 0.25 so both gate regimes occur
    assert w_max.median() > 0.4
    assert (w_max < 0.25).any() and (w_max > 0.9).any()


def test_drift_needle_workload():
    w = wl.scaled(wl.WORKLOADS["long_128k_b4"], seq_len=8192, n_layers=1, batch=1, n_kv_heads=1)
    pos = wl.needle_positions(w, 0, 0, 0, "cpu")
    assert 0.005 < pos.numel() / 8192 < 0.02 and pos.max() < 8192 - 64
    K, _ = wl.unit_kv(w, 0, 0, 0)
    norms = K.float().norm(dim=1)
    assert norms[pos].mean() > 1.3 * norms[torch.ones(8192, dtype=torch.bool).index_fill_(0, pos, False)].mean()


def test_drawn_residual_counts():
    w = wl.WORKLOADS["small_budget_b64"]
    r = w.residual_override()
    assert r.shape == (w.n_units,) and r.min() >= 0 and r.max() <= 64
    per = r.reshape(w.n_layers, w.batch, w.n_kv_heads)
    assert np.all(per == per[:, :1, :])                                  # shared across batch
    frac0 = np.mean(per[:, 0, :] == 0)
    assert 0.05 < frac0 < 0.3


def test_layer_inputs_stack_units():
    w = wl.scaled(wl.WORKLOADS["tiny"], seq_len=512, n_kv_heads=2, batch=2, n_obs=8, n_fit=6, n_val=2)
    K, V, Qo, Qd = wl.layer_inputs(w, 0, "cpu", n_dec_steps=3)
    k, v = wl.unit_kv(w, 0, 1, 1)
    assert torch.equal(K[1, 1], k) and torch.equal(V[1, 1], v)
    qo = wl.unit_obs_queries(w, 0, 1, 1, k)
    assert torch.equal(Qo[1, 4:8], qo)
    qd = wl.unit_decode_queries(w, 0, 1, 1, k, 3)
    assert torch.equal(Qd[:, 1, 4:8], qd.permute(1, 0, 2))
