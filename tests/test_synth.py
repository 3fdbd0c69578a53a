"""The seeded input generator shared by the oracle and the CUDA path: reproducible, thread
independent, rounded to bf16 exactly as the hardware rounds, and shaped as the workloads
state (segments, heavy hitters, ragged lengths, zero rows past each sequence)."""
import numpy as np
import pytest
import torch

import synth


def test_bf16_rounding_matches_torch_round_to_nearest_even():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 10.0 ** rng.integers(-6, 6, 100000),
                        np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -1.0 - 2.0 ** -8, 0.0, -0.0],
                                 dtype=np.float32)])
    want = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(synth.round_bf16(x), want)


def test_generation_is_reproducible_and_thread_independent():
    wl = synth.WORKLOADS["llama_layer"].with_(n=2048, batch=2, ragged=(0.5, 1.0))
    a = synth.gen_layer(wl, 3, threads=1)
    b = synth.gen_layer(wl, 3, threads=8)
    for k in ("K", "V", "Q_obs", "n_len"):
        np.testing.assert_array_equal(a[k], b[k])
    c = synth.gen_layer(wl, 4, threads=1)
    assert not np.array_equal(a["K"], c["K"])  # layers draw their own streams


def test_shapes_ragged_lengths_and_zero_tails():
    wl = synth.WORKLOADS["llama_layer"].with_(n=4096, batch=4, ragged=(0.5, 1.0), seed=7)
    x = synth.gen_layer(wl, 0)
    B, Hkv, Hq, d, W = wl.batch, wl.num_kv_heads, wl.num_q_heads, wl.head_dim, wl.obs_window
    assert x["K"].shape == (B, Hkv, wl.n, d) and x["V"].shape == (B, Hkv, wl.n, d)
    assert x["Q_obs"].shape == (B, Hq, W, d)
    for b, n_b in enumerate(x["n_len"]):
        assert wl.n // 2 <= n_b <= wl.n
        assert not x["K"][b, :, n_b:].any() and not x["V"][b, :, n_b:].any()
        assert np.abs(x["K"][b, :, :n_b]).sum(axis=-1).min() > 0


def test_bf16_workloads_hold_bf16_values():
    wl = synth.WORKLOADS["llama_layer"].with_(n=1024)
    x = synth.gen_layer(wl, 0)
    for k in ("K", "V", "Q_obs"):
        np.testing.assert_array_equal(synth.round_bf16(x[k]), x[k])


def test_segments_heavy_hitters_and_value_similarity():
    """Tiny workload: 64 segments of 16 tokens, sigma 0.3: values of one segment are close
    (cosine near 1), values of different segments are not; the 8 heavy hitters have key rows
    4x the segment-mates' scale and are shared by both KV heads."""
    wl = synth.WORKLOADS["tiny"]
    x = synth.gen_layer(wl, 0)
    V = x["V"][0, 0].astype(np.float64)
    Vn = V / np.linalg.norm(V, axis=1, keepdims=True)
    same = [Vn[16 * s + i] @ Vn[16 * s + j] for s in range(64) for i, j in ((0, 5), (3, 11))]
    other = [Vn[16 * s] @ Vn[16 * (s + 1)] for s in range(63)]
    assert min(same) > 0.8 and np.mean(other) < 0.3
    hh = synth.heavy_positions(wl, 0, 0, wl.n)
    assert len(hh) == 8 and len(set(hh.tolist())) == 8
    Kn = np.linalg.norm(x["K"][0].astype(np.float64), axis=-1)    # [Hkv][n]
    others = np.setdiff1d(np.arange(wl.n), hh)
    assert Kn[:, hh].min() > 2.0 * np.median(Kn[:, others])


@pytest.mark.parametrize("b,n,r", [(1, 8192, 0.1), (8, 32768, 0.25), (64, 131072, 0.5)])
def test_serving_sweep_points(b, n, r):
    wl = synth.sweep(b, n, r)
    assert wl.batch == b and wl.n == n and wl.rho == r and wl.layers == 1 and wl.ragged == (0.5, 1.0)
    n_len = synth.seq_lengths(wl)
    assert n_len.shape == (b,) and (n_len >= n // 2).all() and (n_len <= n).all()
    assert (b, n, r) in synth.SWEEP_POINTS


def test_gen_sequence_equals_the_layers_sequence():
    """A sequence generated alone holds exactly the values gen_layer gives it."""
    wl = synth.sweep(3, 2048, 0.25)
    x = synth.gen_layer(wl, 2, threads=4)
    for b in range(wl.batch):
        s = synth.gen_sequence(wl, 2, b, threads=2)
        n = int(x["n_len"][b])
        assert s["n"] == n
        np.testing.assert_array_equal(s["K"], x["K"][b, :, :n])
        np.testing.assert_array_equal(s["V"], x["V"][b, :, :n])
        np.testing.assert_array_equal(s["Q_obs"], x["Q_obs"][b])
