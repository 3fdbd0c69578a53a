"""Pins for the fp64 oracle: closed forms, hand-worked examples (tests/golden/), library
routines and brute force on tiny inputs, chosen so that a dropped term, a wrong sign or index,
a transposed operand or a wrong tie-break in the oracle fails at least one of them.

CPU only."""
import json
import math
import os

import numpy as np
import pytest
import torch

import synth
from oracle import selkv_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def rng(seed):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- Sec. 3.1: budget
def test_budget_floor_and_recent_window():
    # m = floor(rho n), m_s = m - m_r (Sec. 3.1); 25% of 1024 is 256 entries, 240 by score
    assert O.budget(1024, 0.25, 16) == (256, 240)
    assert O.budget(1023, 0.25, 16) == (255, 239)      # floor, not round
    assert O.budget(100000, 0.25, 16) == (25000, 24984)
    assert O.budget(40, 0.25, 16) == (10, -6)          # below the recent window: invalid


# ---------------------------------------------------------------- Sec. 3.1 re-pass
def test_uniform_keys_closed_form():
    """With all keys equal every visible score ties, so row i spreads 1/(p_i+1) over
    j <= p_i = n-W+i.  Then a_j = H_n - H_max(j, n-W) (harmonic numbers): this pins the
    causal direction, the window's positions and the average over the query group."""
    n, W, d, Hq, Hkv = 50, 8, 4, 4, 2
    Q = rng(1).standard_normal((Hq, W, d))
    K = np.ones((Hkv, n, d))
    a = O.cumulative_attention(Q, K, n)
    H = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, n + 1))])
    expect = np.array([H[n] - H[max(j, n - W)] for j in range(n)])
    for kv in range(Hkv):
        np.testing.assert_allclose(a[kv], expect, rtol=1e-13, atol=1e-15)
    assert abs(a.sum(axis=1) - W).max() < 1e-12      # each window row carries mass 1


def test_observation_attention_matches_torch_sdpa():
    """Library pin: torch SDPA in fp64 with identity values returns the attention matrix
    itself (default scale 1/sqrt(d), boolean mask True = visible)."""
    n, W, d, Hq, Hkv = 37, 6, 8, 4, 2
    r = rng(2)
    Q = r.standard_normal((Hq, W, d)) * 2
    K = r.standard_normal((Hkv, n, d))
    A = O.observation_attention(Q, K, n)
    G = Hq // Hkv
    pos = n - W + np.arange(W)
    mask = torch.from_numpy(np.arange(n)[None, :] <= pos[:, None])
    for h in range(Hq):
        out = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(Q[h])[None], torch.from_numpy(K[h // G, :n])[None],
            torch.eye(n, dtype=torch.float64)[None], attn_mask=mask[None])
        np.testing.assert_allclose(A[h], out[0].numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(A.sum(axis=2), 1.0, rtol=1e-13)


def test_cumulative_attention_brute_force():
    n, W, d, Hq, Hkv = 12, 3, 2, 4, 2
    r = rng(3)
    Q, K = r.standard_normal((Hq, W, d)), r.standard_normal((Hkv, n, d))
    G = Hq // Hkv
    a = O.cumulative_attention(Q, K, n)
    brute = np.zeros((Hkv, n))
    for h in range(Hq):
        for i in range(W):
            p = n - W + i
            logits = [sum(Q[h, i, t] * K[h // G, j, t] for t in range(d)) / math.sqrt(d)
                      for j in range(p + 1)]
            mx = max(logits)
            w = [math.exp(x - mx) for x in logits]
            z = sum(w)
            for j in range(p + 1):
                brute[h // G, j] += w[j] / z / G
    np.testing.assert_allclose(a, brute, rtol=1e-12)


# ---------------------------------------------------------------- Eq. 1 + pooling
def test_contribution_score_is_attention_times_value_norm():
    a = np.array([[0.5, 2.0, 0.0]])
    V = np.array([[[3.0, 4.0], [1.0, 0.0], [7.0, 7.0]]])
    np.testing.assert_allclose(O.contribution_scores(a, V, 3), [[2.5, 2.0, 0.0]])


def test_pool_impulse_and_edges():
    n_cand, k = 10, 5
    c = np.zeros((1, 14))
    c[0, 4] = 1.0
    np.testing.assert_allclose(O.pool_scores(c, n_cand, k)[0],
                               [0, 0, .2, .2, .2, .2, .2, 0, 0, 0], atol=1e-15)
    c = np.zeros((1, 14))
    c[0, 9] = 1.0          # last candidate: only the left neighbours see it
    c[0, 10:] = 100.0      # recent window: never pooled in
    np.testing.assert_allclose(O.pool_scores(c, n_cand, k)[0],
                               [0, 0, 0, 0, 0, 0, 0, .2, .2, .2], atol=1e-15)
    ones = np.ones((1, n_cand))
    np.testing.assert_allclose(O.pool_scores(ones, n_cand, 5)[0],
                               [.6, .8, 1, 1, 1, 1, 1, 1, .8, .6], atol=1e-15)


# ---------------------------------------------------------------- Eq. 2 + Sec. 3.3
def test_top_k_brute_force_with_ties():
    r = rng(4)
    for trial in range(200):
        n = int(r.integers(1, 30))
        vals = r.integers(0, 5, size=n).astype(float)    # many ties
        k = int(r.integers(0, n + 1))
        chosen, left = [], list(range(n))
        for _ in range(k):                               # repeated argmax, lowest index
            best = left[0]
            for j in left[1:]:
                if vals[j] > vals[best]:
                    best = j
            chosen.append(best)
            left.remove(best)
        expect = np.zeros(n, dtype=bool)
        expect[chosen] = True
        assert (O.top_k_mask(vals, k) == expect).all()


def test_union_trim_worked_example():
    gd = golden("union_trim.json")
    cp = np.array(gd["c_pooled"], dtype=float)
    sel = O.select_shared(cp, gd["n"], gd["m_s"], gd["recent"])
    for kv, expect in enumerate(gd["per_kv"]):
        assert np.flatnonzero(sel.per_kv[kv]).tolist() == expect
    assert np.flatnonzero(sel.union).tolist() == gd["union"]
    assert sel.trimmed
    assert np.flatnonzero(sel.kept).tolist() == gd["kept"]


def test_union_without_trim_is_shared_topk():
    cp = np.array([[3, 1, 2, 0], [3, 0, 2, 1]], dtype=float)
    sel = O.select_shared(cp, 6, 2, 2)
    assert not sel.trimmed
    assert np.flatnonzero(sel.kept).tolist() == [0, 2, 4, 5]


# ---------------------------------------------------------------- Eq. 3
def test_routing_worked_example():
    gd = golden("routing.json")
    n, B = gd["n"], gd["bucket"]
    kept = np.zeros(n, dtype=bool)
    kept[gd["kept"]] = True
    a = np.full(n, 0.01)
    for k, v in gd["a"].items():
        a[int(k)] = v
    t = O.route(a, kept, B, O.EMPTY_EXPAND)
    expect = {int(k): v for k, v in gd["expand"].items()}
    for j in range(n):
        assert t[j] == (expect[j] if j in expect else -1), j
    t = O.route(a, kept, B, O.EMPTY_DROP)
    for j in range(n):
        if j in gd["drop_policy_untargeted"] or kept[j]:
            assert t[j] == -1
        else:
            assert t[j] == expect[j]


def test_routing_brute_force():
    """Explicit scan: for each evicted j, the kept i of the nearest non-empty ring of
    buckets with the largest a (lowest index on ties)."""
    r = rng(5)
    for trial in range(30):
        n, B = int(r.integers(8, 90)), int(r.integers(2, 9))
        kept = r.random(n) < 0.15
        kept[-1] = True
        a = r.integers(1, 6, size=n).astype(float)
        t = O.route(a, kept, B, O.EMPTY_EXPAND)
        for j in range(n):
            if kept[j]:
                assert t[j] == -1
                continue
            best = None
            for dist in range(n):
                cands = [i for i in range(n) if kept[i] and abs(i // B - j // B) == dist]
                if cands:
                    best = min(cands, key=lambda i: (-a[i], i))
                    break
            assert t[j] == best


# ---------------------------------------------------------------- Eq. 4-6, Sec. 3.5-3.6
def test_gate_merge_ratio_worked_example():
    gd = golden("gate_merge.json")
    V = np.array([gd["v_target"]] + gd["contributors"], dtype=float)
    a = np.array([gd["a_target"]] + gd["a_contrib"])
    target = np.array([-1] + [0] * len(gd["contributors"]))
    g, sim, dec = O.gate(V, target, O.GATE_COSINE)
    np.testing.assert_allclose(g[1:], gd["g"], atol=1e-15)
    assert dec[1:].tolist() == gd["decision"]
    Vm, R = O.merge(a, V, np.array([0]), target, g)
    np.testing.assert_allclose(Vm[0], gd["v_merged"], rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(R[0], gd["R"], rtol=1e-14)
    np.testing.assert_allclose(O.gqa_bias(R[None], 0.5)[0], gd["bias"], rtol=1e-14)


def test_gqa_bias_is_log_of_mean_ratio():
    gd = golden("gqa_bias.json")
    np.testing.assert_allclose(O.gqa_bias(np.array(gd["R"]), gd["alpha"]), gd["bias"],
                               rtol=1e-14, atol=1e-16)


def test_gate_modes():
    V = np.array([[1.0, 0], [-1.0, 0], [0.6, 0.8]])
    t = np.array([-1, 0, 0])
    assert O.gate(V, t, O.GATE_OPEN)[0].tolist() == [0, 1, 1]
    assert O.gate(V, t, O.GATE_CLOSED)[0].tolist() == [0, 0, 0]
    np.testing.assert_allclose(O.gate(V, t, O.GATE_COSINE)[0], [0, 0, 0.6])


# ---------------------------------------------------------------- whole pipeline
def _tiny(seed=0, **kw):
    wl = synth.WORKLOADS["tiny"].with_(seed=seed, **kw)
    x = synth.gen_layer(wl, 0)
    n = int(x["n_len"][0])
    return wl, x["K"][0].astype(float), x["V"][0].astype(float), x["Q_obs"][0].astype(float), n


def test_gate_closed_is_pure_eviction():
    """g = 0 everywhere reduces Eq. 5 to dropping (Sec. 3.5; ablation 'eviction only')."""
    wl, K, V, Q, n = _tiny()
    r = O.compress(K, V, Q, n, wl.rho, O.Params(gate_mode=O.GATE_CLOSED))
    # (a_i v_i) / a_i is v_i up to one rounding of fp64
    np.testing.assert_allclose(r.V_c, V[:, r.kept_idx], rtol=1e-15, atol=0)
    np.testing.assert_array_equal(r.K_c, K[:, r.kept_idx])
    np.testing.assert_array_equal(r.R, 1.0)
    np.testing.assert_array_equal(r.bias, 0.0)
    assert (r.decision[r.target >= 0] == O.DECISION_DROP).all()


def test_gate_open_is_attention_weighted_merge():
    """g = 1 reduces Eq. 5 to the attention-weighted average of each kept token and the
    tokens routed to it (Sec. 3.5; ablation 'merge all'), computed here by explicit scans."""
    wl, K, V, Q, n = _tiny(seed=1)
    r = O.compress(K, V, Q, n, wl.rho, O.Params(gate_mode=O.GATE_OPEN))
    for kv in range(K.shape[0]):
        for s, i in enumerate(r.kept_idx):
            group = [i] + [j for j in range(n) if r.target[kv, j] == i]
            w = np.array([r.a[kv, j] for j in group])
            expect = sum(w[t] * V[kv, j] for t, j in enumerate(group)) / w.sum()
            np.testing.assert_allclose(r.V_c[kv, s], expect, rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(r.R[kv, s], w.sum() / r.a[kv, i], rtol=1e-12)


def test_full_budget_is_full_attention():
    """rho = 1 evicts nothing: the cache is unchanged, R = 1, bias = 0, and decode is
    exact full attention (checked against torch SDPA in fp64)."""
    wl, K, V, Q, n = _tiny(seed=2)
    r = O.compress(K, V, Q, n, 1.0)
    assert r.kept_idx.tolist() == list(range(n))
    np.testing.assert_allclose(r.V_c, V[:, :n], rtol=1e-15, atol=0)
    np.testing.assert_array_equal(r.bias, 0.0)
    q = rng(6).standard_normal((wl.num_q_heads, wl.head_dim))
    out = O.decode(q, r.K_c, r.V_c, r.bias, n)
    G = wl.group
    for h in range(wl.num_q_heads):
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[h])[None, None], torch.from_numpy(K[h // G, :n])[None],
            torch.from_numpy(V[h // G, :n])[None])
        np.testing.assert_allclose(out[h], ref[0, 0].numpy(), rtol=1e-11, atol=1e-13)


def test_decode_bias_matches_sdpa_additive_mask():
    r = rng(7)
    Hq, Hkv, L, d = 4, 2, 23, 8
    q = r.standard_normal((Hq, d))
    Kc, Vc = r.standard_normal((Hkv, L, d)), r.standard_normal((Hkv, L, d))
    bias = r.random(L) * 2
    out = O.decode(q, Kc, Vc, bias, L)
    for h in range(Hq):
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[h])[None, None], torch.from_numpy(Kc[h // 2])[None],
            torch.from_numpy(Vc[h // 2])[None], attn_mask=torch.from_numpy(bias)[None, None])
        np.testing.assert_allclose(out[h], ref[0, 0].numpy(), rtol=1e-12, atol=1e-14)


def test_merged_duplicates_recover_softmax_mass():
    """m identical tokens merged into one kept copy with g = 1 and equal attention give
    R = m; with alpha = 1 the bias is ln m and decode over the compressed cache equals decode
    over the full cache exactly (the attention-sag correction of Sec. 3.6)."""
    r = rng(8)
    Hq, Hkv, W, d, n, B = 2, 1, 4, 8, 64, 32
    K = r.standard_normal((Hkv, n, d))
    V = r.standard_normal((Hkv, n, d))
    dup = list(range(40, 45))                   # 5 identical tokens in bucket 1
    K[:, dup] = K[:, dup[:1]]
    V[:, dup] = V[:, dup[:1]]
    Q = r.standard_normal((Hq, W, d))
    kept = np.ones(n, dtype=bool)
    kept[dup[1:]] = False                       # keep the first copy only
    rho = kept.sum() / n
    target = np.full((Hkv, n), -1)
    target[:, dup[1:]] = dup[0]                 # the copies route to their kept twin
    res = O.compress(K, V, Q, n, rho, O.Params(alpha=1.0, recent=0, bucket=B),
                     follow_kept=kept, follow_target=target)
    s = int(np.flatnonzero(res.kept_idx == dup[0])[0])
    np.testing.assert_allclose(res.g[0, dup[1:]], 1.0, rtol=1e-15)
    np.testing.assert_allclose(res.R[0, s], len(dup), rtol=1e-13)
    np.testing.assert_allclose(res.bias[s], math.log(len(dup)), rtol=1e-13)
    others = np.delete(np.arange(res.kept_idx.size), s)
    np.testing.assert_allclose(res.bias[others], 0.0, atol=1e-15)
    q = r.standard_normal((Hq, d))
    full = O.decode(q, K, V, None, n)
    comp = O.decode(q, res.K_c, res.V_c, res.bias, res.kept_idx.size)
    np.testing.assert_allclose(comp, full, rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("seed,dtype", [(0, "fp32"), (3, "bf16")])
def test_pipeline_invariants(seed, dtype):
    wl, K, V, Q, n = _tiny(seed=seed, dtype=dtype)
    p = O.Params()
    r = O.compress(K, V, Q, n, wl.rho, p)
    m, m_s = O.budget(n, wl.rho, p.recent)
    assert r.kept_idx.size == m and (np.diff(r.kept_idx) > 0).all()
    assert set(range(n - p.recent, n)) <= set(r.kept_idx.tolist())
    assert int(r.sel.kept_cand.sum()) == m_s
    Hkv = K.shape[0]
    for kv in range(Hkv):
        ev = np.flatnonzero(~r.sel.kept)
        t = r.target[kv, ev]
        assert (t >= 0).all()                                 # everyone has a target
        assert r.sel.kept[t].all()
        nonempty = np.array([r.sel.kept[(j // p.bucket) * p.bucket:
                                        (j // p.bucket + 1) * p.bucket].any() for j in ev])
        assert (t[nonempty] // p.bucket == ev[nonempty] // p.bucket).all()
        assert (r.R[kv] >= 1.0 - 1e-15).all()
        contributed = np.zeros(r.kept_idx.size, dtype=bool)
        slot = {int(i): s for s, i in enumerate(r.kept_idx)}
        for j in ev:
            if r.g[kv, j] > 0:
                contributed[slot[int(r.target[kv, j])]] = True
        assert (r.R[kv][~contributed] == 1.0).all()
        lhs = (r.a[kv, r.kept_idx] * r.R[kv]).sum()            # mass conservation
        rhs = r.a[kv, r.kept_idx].sum() + (r.g[kv, ev] * r.a[kv, ev]).sum()
        assert abs(lhs - rhs) <= 1e-12 * rhs
        for s, i in enumerate(r.kept_idx):                     # convex hull
            members = [i] + [j for j in ev if r.target[kv, j] == i and r.g[kv, j] > 0]
            lo, hi = V[kv, members].min(axis=0), V[kv, members].max(axis=0)
            assert (r.V_c[kv, s] >= lo - 1e-12).all() and (r.V_c[kv, s] <= hi + 1e-12).all()
    q = rng(9).standard_normal((wl.num_q_heads, wl.head_dim))
    r0 = O.compress(K, V, Q, n, wl.rho, O.Params(alpha=0.0))
    np.testing.assert_array_equal(r0.bias, 0.0)                 # alpha = 0: no compensation
    np.testing.assert_allclose(O.decode(q, r0.K_c, r0.V_c, r0.bias, m),
                               O.decode(q, r0.K_c, r0.V_c, None, m), rtol=1e-14, atol=1e-15)


def test_follow_mode_reproduces_own_choices():
    wl, K, V, Q, n = _tiny(seed=4)
    r = O.compress(K, V, Q, n, wl.rho)
    f = O.compress(K, V, Q, n, wl.rho, follow_per_kv=r.sel.per_kv, follow_kept=r.sel.kept,
                   follow_target=r.target)
    np.testing.assert_array_equal(f.V_c, r.V_c)
    np.testing.assert_array_equal(f.bias, r.bias)


def test_rejects_budget_below_recent_window():
    wl, K, V, Q, n = _tiny()
    with pytest.raises(ValueError):
        O.compress(K, V, Q, n, 0.01)


# ---------------------------------------------------------------- per-head mode (Sec. 3.3, 3.6)
def test_per_head_bias_worked_example():
    gd = golden("per_head_bias.json")
    np.testing.assert_allclose(O.per_head_bias(np.array(gd["R"]), gd["alpha"]), gd["bias"],
                               rtol=1e-14, atol=1e-16)


def _mha(seed, Hkv=4, n=640, d=32, W=16):
    r = rng(seed)
    K = r.standard_normal((Hkv, n, d))
    V = r.standard_normal((Hkv, n, d))
    Q = r.standard_normal((Hkv, W, d)) * 1.5   # G = 1: one query head per KV head
    return K, V, Q, n


def test_per_head_selection_brute_force():
    """Eq. 2 per head: each head's kept set is the recent window plus its m_s best pooled
    scores, checked against a full sort with the (value desc, position asc) key."""
    K, V, Q, n = _mha(11)
    p = O.Params(select_mode=O.SELECT_PER_HEAD, recent=8, bucket=16)
    r = O.compress(K, V, Q, n, 0.25, p)
    n_cand = n - p.recent
    for kv in range(K.shape[0]):
        order = sorted(range(n_cand), key=lambda j: (-r.c_pooled[kv, j], j))
        expect = sorted(order[:r.m_s]) + list(range(n_cand, n))
        assert r.kept_idx[kv].tolist() == expect


def test_per_head_with_one_kv_head_equals_shared():
    """With a single KV head the union of one set is that set and no trim happens, so both
    modes must give the same cache, targets and bias (Sec. 3.3, Sec. 3.6)."""
    K, V, Q, n = _mha(12, Hkv=1)
    shared = O.compress(K, V, Q, n, 0.25, O.Params(recent=8, bucket=16))
    per = O.compress(K, V, Q, n, 0.25, O.Params(recent=8, bucket=16, select_mode=O.SELECT_PER_HEAD))
    assert per.kept_idx[0].tolist() == shared.kept_idx.tolist()
    np.testing.assert_array_equal(per.target, shared.target)
    np.testing.assert_array_equal(per.V_c, shared.V_c)
    np.testing.assert_array_equal(per.K_c, shared.K_c)
    np.testing.assert_allclose(per.bias[0], shared.bias, rtol=0, atol=0)


def test_per_head_sets_differ_and_follow_their_heads():
    """Heads whose attention favours different positions keep different sets, each with its
    own favoured positions (the point of per-head selection, Sec. 3.3)."""
    K, V, Q, n = _mha(13, Hkv=2)
    hot = {0: [40, 41, 300], 1: [120, 121, 500]}
    for kv, pos in hot.items():
        for j in pos:
            K[kv, j] = 6.0 * Q[kv].mean(axis=0) / np.linalg.norm(Q[kv].mean(axis=0))
    r = O.compress(K, V, Q, n, 0.1, O.Params(select_mode=O.SELECT_PER_HEAD, recent=8, bucket=16))
    s0, s1 = set(r.kept_idx[0].tolist()), set(r.kept_idx[1].tolist())
    assert s0 != s1
    assert set(hot[0]) <= s0 and set(hot[1]) <= s1


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_per_head_pipeline_invariants(seed):
    """Per head: exactly m kept, recent window kept, every target a kept token of that head
    in the evicted token's bucket when that bucket has one, R >= 1, mass conservation
    sum_S a_i R_i = sum_S a_i + sum_E g_j a_j, and a closed gate is pure eviction."""
    K, V, Q, n = _mha(20 + seed)
    p = O.Params(select_mode=O.SELECT_PER_HEAD, recent=8, bucket=16)
    r = O.compress(K, V, Q, n, 0.3, p)
    for kv in range(K.shape[0]):
        kept = r.kept_idx[kv]
        assert kept.size == r.m and set(range(n - p.recent, n)) <= set(kept.tolist())
        ks = set(kept.tolist())
        for j in range(n):
            t = int(r.target[kv, j])
            if j in ks:
                assert t == -1
                continue
            assert t in ks
            same = [i for i in kept if i // p.bucket == j // p.bucket]
            if same:
                assert t // p.bucket == j // p.bucket
        assert (r.R[kv] >= 1.0 - 1e-15).all()
        lhs = float((r.a[kv, kept] * r.R[kv]).sum())
        ev = r.target[kv] >= 0
        rhs = float(r.a[kv, kept].sum() + (r.g[kv, ev] * r.a[kv, ev]).sum())
        assert abs(lhs - rhs) <= 1e-12 * rhs
        np.testing.assert_allclose(r.bias[kv], p.alpha * np.log(r.R[kv]), rtol=0, atol=0)
    closed = O.compress(K, V, Q, n, 0.3, O.Params(select_mode=O.SELECT_PER_HEAD, recent=8, bucket=16,
                                                  gate_mode=O.GATE_CLOSED))
    for kv in range(K.shape[0]):
        np.testing.assert_allclose(closed.V_c[kv], V[kv, closed.kept_idx[kv]], rtol=1e-15, atol=0)
    np.testing.assert_array_equal(closed.bias, 0.0)


# ---------------------------------------------------------------- Eq. 7: RoPE repositioning
@pytest.mark.parametrize("layout,key", [(O.ROPE_HALF, "half"), (O.ROPE_INTERLEAVED, "interleaved")])
def test_rope_reposition_worked_example(layout, key):
    gd = golden("rope_reposition.json")
    got = O.rope(O.rope_inverse(np.array(gd["k"]), gd["p_old"], gd["theta"], layout), gd["p_new"],
                 gd["theta"], layout)
    np.testing.assert_allclose(got, gd[key], rtol=1e-14, atol=1e-15)
    out = O.reposition(np.array([[9.0, 9, 9, 9], gd["k"]]), np.array([0, gd["p_old"]]), gd["theta"], layout)
    np.testing.assert_allclose(out[1], gd[key], rtol=1e-14, atol=1e-15)   # slot 1 = p_new
    np.testing.assert_allclose(out[0], [9.0, 9, 9, 9], rtol=0, atol=1e-15)  # no move: unchanged


@pytest.mark.parametrize("layout", [O.ROPE_HALF, O.ROPE_INTERLEAVED])
def test_rope_reposition_equals_embedding_at_new_position(layout):
    """A key embedded at p_old and repositioned equals the raw key embedded at p_new,
    computed independently with complex exponentials: (x + i y) e^{i p w_f}."""
    r = rng(31)
    d, theta = 16, 10000.0
    raw = r.standard_normal((5, d))
    p_old = np.array([3, 17, 400, 9999, 123456])
    w = theta ** (-2.0 * np.arange(d // 2) / d)
    xi, yi = O.rope_pairs(d, layout)

    def embed(k, p):
        z = (k[xi] + 1j * k[yi]) * np.exp(1j * p * w)
        out = np.empty(d)
        out[xi], out[yi] = z.real, z.imag
        return out
    K = np.stack([embed(raw[i], p_old[i]) for i in range(5)])
    got = O.reposition(K, p_old, theta, layout)
    want = np.stack([embed(raw[s], s) for s in range(5)])
    np.testing.assert_allclose(got, want, rtol=1e-9, atol=1e-9)
    np.testing.assert_allclose(np.linalg.norm(got, axis=1), np.linalg.norm(K, axis=1), rtol=1e-13)


def test_rope_scores_depend_on_relative_position():
    """q . k after RoPE depends only on the position difference, so a query at new position
    t_new scores a repositioned key exactly as a query at t_new + (p_old - p_new) scored the
    original (the property repositioning relies on)."""
    r = rng(32)
    d, theta = 8, 500.0
    q, k = r.standard_normal(d), r.standard_normal(d)
    for layout in (O.ROPE_HALF, O.ROPE_INTERLEAVED):
        k_old = O.rope(k, 50, theta, layout)
        k_new = O.reposition(np.stack([np.zeros(d), np.zeros(d), k_old]), np.array([0, 1, 50]), theta, layout)[2]
        s_new = O.rope(q, 10, theta, layout) @ k_new          # query 8 positions after slot 2
        s_old = O.rope(q, 58, theta, layout) @ k_old          # the same distance in the old frame
        assert abs(s_new - s_old) < 1e-12


def test_compress_with_rope_keeps_values_and_rotates_keys():
    wl, K, V, Q, n = _tiny(seed=3)
    base = O.compress(K, V, Q, n, wl.rho)
    rot = O.compress(K, V, Q, n, wl.rho, O.Params(rope=O.ROPE_HALF, rope_theta=10000.0))
    np.testing.assert_array_equal(rot.V_c, base.V_c)
    np.testing.assert_array_equal(rot.bias, base.bias)
    for kv in range(K.shape[0]):
        np.testing.assert_allclose(rot.K_c[kv], O.reposition(K[kv, base.kept_idx], base.kept_idx,
                                                             10000.0, O.ROPE_HALF), rtol=0, atol=0)
        np.testing.assert_allclose(np.linalg.norm(rot.K_c[kv], axis=1), np.linalg.norm(base.K_c[kv], axis=1),
                                   rtol=1e-12)


# ---------------------------------------------------------------- count bias (KeepKV, Sec. 3.6)
def test_count_bias_worked_example():
    """Hand-worked: kept tokens 0 and 3; tokens 1, 2 routed to 0 with g = 0.5 and 0 (only one
    merges), token 4 routed to 3 with g = 1: M = (1, 1) for this head; with a second head
    where M = (3, 0), the shared bias is ln(1 + 2) and ln(1 + 0.5); per head it is ln 2, ln 2
    and ln 4, ln 1 (alpha = 1, KeepKV's log(1 + M))."""
    kept = np.array([0, 3])
    target = np.array([-1, 0, 0, -1, 3])
    g = np.array([0.0, 0.5, 0.0, 0.0, 1.0])
    M0 = O.merge_counts(kept, target, g)
    assert M0.tolist() == [1.0, 1.0]
    M = np.stack([M0, np.array([3.0, 0.0])])
    np.testing.assert_allclose(O.count_bias(M, 1.0, per_head=False), [math.log(3.0), math.log(1.5)], rtol=1e-15)
    np.testing.assert_allclose(O.count_bias(M, 1.0, per_head=True),
                               [[math.log(2.0), math.log(2.0)], [math.log(4.0), 0.0]], rtol=1e-15)


def test_count_bias_compress_matches_explicit_counts():
    wl, K, V, Q, n = _tiny(seed=4)
    for mode in (O.SELECT_SHARED, O.SELECT_PER_HEAD):
        r = O.compress(K, V, Q, n, wl.rho, O.Params(bias_mode=O.BIAS_COUNT, select_mode=mode))
        Hkv = K.shape[0]
        kept = r.kept_idx if mode == O.SELECT_PER_HEAD else np.stack([r.kept_idx] * Hkv)
        M = np.array([[sum(1 for j in range(n) if r.target[kv, j] == i and r.g[kv, j] > 0) for i in kept[kv]]
                      for kv in range(Hkv)], dtype=float)
        want = 0.5 * np.log(1.0 + (M if mode == O.SELECT_PER_HEAD else M.mean(axis=0)))
        np.testing.assert_allclose(r.bias, want, rtol=1e-14, atol=0)
        closed = O.compress(K, V, Q, n, wl.rho, O.Params(bias_mode=O.BIAS_COUNT, select_mode=mode,
                                                          gate_mode=O.GATE_CLOSED))
        np.testing.assert_array_equal(closed.bias, 0.0)   # nothing merges, so no count


# ---------------------------------------------------------------- full cosine routing (Sec. 3.4)
def test_cosine_routing_worked_example():
    """Hand-worked: kept tokens 0 (v = (1, 0)) and 2 (v = (0, 1)); token 1 = (1, 1) ties
    (cos 1/sqrt 2 with both) and goes to the lower position 0; token 3 = (-1, 3) is closer to
    (0, 1); token 4 = (0, 0) has cosine 0 with both and goes to 0."""
    V = np.array([[1.0, 0], [1, 1], [0, 1], [-1, 3], [0, 0]])
    kept = np.array([True, False, True, False, False])
    assert O.route_cosine(V, kept).tolist() == [-1, 0, -1, 2, 0]


def test_cosine_routing_brute_force():
    r = rng(41)
    n, d = 120, 8
    V = r.standard_normal((n, d))
    V[7] = 0.0
    kept = np.zeros(n, dtype=bool)
    kept[r.choice(n, 30, replace=False)] = True
    t = O.route_cosine(V, kept)
    for j in range(n):
        if kept[j]:
            assert t[j] == -1
            continue
        best, bi = -2.0, -1
        for i in range(n):
            if not kept[i]:
                continue
            den = math.sqrt(float(V[j] @ V[j])) * math.sqrt(float(V[i] @ V[i]))
            c = float(V[j] @ V[i]) / den if den > 0 else 0.0
            if c > best:
                best, bi = c, i
        assert t[j] == bi


def test_cosine_routing_gate_is_the_max_cosine():
    """With cosine routing the gate of j is its largest cosine to any kept token, clamped."""
    wl, K, V, Q, n = _tiny(seed=5)
    r = O.compress(K, V, Q, n, wl.rho, O.Params(routing=O.ROUTE_COSINE))
    ki = r.kept_idx
    for kv in range(K.shape[0]):
        Vk = V[kv, ki]
        nk = np.linalg.norm(Vk, axis=1)
        for j in np.flatnonzero(r.target[kv] >= 0)[:60]:
            cos = (Vk @ V[kv, j]) / (nk * np.linalg.norm(V[kv, j]))
            assert abs(r.g[kv, j] - min(max(cos.max(), 0.0), 1.0)) < 1e-12
        ev = r.target[kv] >= 0
        lhs = float((r.a[kv, ki] * r.R[kv]).sum())
        rhs = float(r.a[kv, ki].sum() + (r.g[kv, ev] * r.a[kv, ev]).sum())
        assert abs(lhs - rhs) <= 1e-12 * rhs      # mass conservation holds for any routing


# ---------------------------------------------------------------- compensation averaged across layers
def test_layer_average_bias_worked_example():
    """Hand-worked, n = 4, two layers: layer 0 keeps positions 0 and 2 with R = 2 and 4, layer 1
    keeps 2 and 3 with R = 2 and 3.  Per position the mean over layers (R = 1 where a layer
    evicted it): 0 -> (2 + 1) / 2 = 1.5, 2 -> (4 + 2) / 2 = 3, 3 -> (1 + 3) / 2 = 2."""
    out = O.layer_average_bias([np.array([2.0, 4.0]), np.array([2.0, 3.0])],
                               [np.array([0, 2]), np.array([2, 3])], 4, 0.5, count=False)
    np.testing.assert_allclose(out[0], 0.5 * np.log([1.5, 3.0]), rtol=0, atol=1e-15)
    np.testing.assert_allclose(out[1], 0.5 * np.log([3.0, 2.0]), rtol=0, atol=1e-15)
    # the count variant: M = 0 where evicted, bias = alpha ln(1 + mean M)
    out = O.layer_average_bias([np.array([2.0, 4.0]), np.array([2.0, 3.0])],
                               [np.array([0, 2]), np.array([2, 3])], 4, 1.0, count=True)
    np.testing.assert_allclose(out[0], np.log([2.0, 4.0]), rtol=0, atol=1e-15)   # 1 + 1, 1 + 3
    np.testing.assert_allclose(out[1], np.log([4.0, 2.5]), rtol=0, atol=1e-15)   # 1 + 3, 1 + 1.5


def test_layer_average_bias_reductions():
    """One layer, or identical layers, give back the per-layer bias (Sec. 3.6, R16 / R19); the
    result does not depend on the order of the layers; per-head shapes average per head."""
    r = rng(51)
    n, m, Hkv = 300, 80, 3
    kept = np.sort(r.choice(n, m, replace=False))
    R = 1.0 + r.exponential(1.0, size=m)
    np.testing.assert_allclose(O.layer_average_bias([R], [kept], n, 0.5, False)[0], 0.5 * np.log(R), atol=1e-15)
    for out in O.layer_average_bias([R, R, R], [kept, kept, kept], n, 0.5, False):
        np.testing.assert_allclose(out, 0.5 * np.log(R), atol=1e-14)
    layers = [(1.0 + r.exponential(1.0, size=m), np.sort(r.choice(n, m, replace=False))) for _ in range(4)]
    a = O.layer_average_bias([q for q, _ in layers], [k for _, k in layers], n, 0.5, False)
    perm = [2, 0, 3, 1]
    b = O.layer_average_bias([layers[i][0] for i in perm], [layers[i][1] for i in perm], n, 0.5, False)
    for i, pi in enumerate(perm):
        np.testing.assert_allclose(b[i], a[pi], atol=1e-14)
    Rh = [1.0 + r.exponential(1.0, size=(Hkv, m)) for _ in range(2)]
    Kh = [np.sort(np.stack([r.choice(n, m, replace=False) for _ in range(Hkv)]), axis=1) for _ in range(2)]
    out = O.layer_average_bias(Rh, Kh, n, 0.5, False)
    for h in range(Hkv):
        want = O.layer_average_bias([Rh[0][h], Rh[1][h]], [Kh[0][h], Kh[1][h]], n, 0.5, False)
        np.testing.assert_allclose(out[0][h], want[0], atol=1e-15)
        np.testing.assert_allclose(out[1][h], want[1], atol=1e-15)
