"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the same seeded
inputs.  Selections, routing targets and merge/drop decisions must agree exactly up to the
near-tie rule of tests/parity.py; continuous outputs within the stated tolerances."""
import numpy as np
import pytest
import torch

import synth
from oracle import selkv_oracle as O
from paper_2607_16213_gb300 import api
import paper_2607_16213_gb300 as S

from parity import (BIAS_ATOL, Stats, check_decode, check_sequence, params_of, run_compress, to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16213_gb300 import build as b
    b.build()
    S.library()


# Small workloads that still span several 64-wide tiles, several buckets and ragged tails.
SMALL = {
    "tiny": synth.WORKLOADS["tiny"],
    "bf16_ragged": synth.WORKLOADS["llama_layer"].with_(name="bf16_ragged", batch=3, n=3001,
                                                        num_q_heads=8, num_kv_heads=2,
                                                        ragged=(0.5, 1.0), seed=11),
    "bf16_d64_g4": synth.WORKLOADS["llama_layer"].with_(name="bf16_d64_g4", batch=2, n=2500,
                                                        head_dim=64, num_q_heads=16,
                                                        num_kv_heads=4, obs_window=40, seed=12),
    "fp32_d128": synth.WORKLOADS["tiny"].with_(name="fp32_d128", head_dim=128, n=1500, batch=2,
                                               ragged=(0.6, 1.0), seed=13),
    # wide GQA groups: G W = 512 rows (two 256-row halves in the column-sum pass) and 384 rows
    # (a half of 128), d 64
    "bf16_g8_w64": synth.WORKLOADS["llama_layer"].with_(name="bf16_g8_w64", batch=2, n=2900,
                                                        num_q_heads=16, num_kv_heads=2,
                                                        ragged=(0.6, 1.0), seed=14),
    "bf16_g16_w24_d64": synth.WORKLOADS["llama_layer"].with_(name="bf16_g16_w24_d64", batch=2, n=2100,
                                                             head_dim=64, num_q_heads=32,
                                                             num_kv_heads=2, obs_window=24,
                                                             ragged=(0.7, 1.0), seed=15),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_compress_parity_small(name):
    wl = SMALL[name]
    x = synth.gen_layer(wl, 0)
    p = O.Params()
    _, host, _ = run_compress(wl, x, p)
    st = Stats()
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p, stats=st)
    print(name, dict(st))


@pytest.mark.parametrize("gate_mode", [O.GATE_OPEN, O.GATE_CLOSED])
def test_compress_gate_end_points(gate_mode):
    wl = SMALL["bf16_ragged"]
    x = synth.gen_layer(wl, 1)
    p = O.Params(gate_mode=gate_mode)
    _, host, _ = run_compress(wl, x, p)
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p)
        m = int(host["lengths"][b])
        if gate_mode == O.GATE_CLOSED:   # pure eviction: V_c = V[S] exactly, R = 1, bias = 0
            kept = host["kept_idx"][b, :m]
            np.testing.assert_array_equal(host["V_c"][b, :, :m], x["V"][b][:, kept])
            np.testing.assert_array_equal(host["ratio"][b, :, :m], 1.0)
            np.testing.assert_array_equal(host["bias"][b, :, :m], 0.0)


@pytest.mark.parametrize("case", [
    dict(rho=1.0),                                   # nothing evicted
    dict(rho=16 / 3001 + 1e-9),                      # m_s = 0: only the recent window
    dict(p=dict(empty_bucket=O.EMPTY_DROP), rho=0.1),
    dict(p=dict(bucket=16, pool_kernel=3, recent=0)),
    dict(p=dict(bucket=7, pool_kernel=1, recent=5, alpha=1.0)),
    dict(p=dict(alpha=0.0)),
])
def test_compress_edge_cases(case):
    wl = SMALL["bf16_ragged"].with_(batch=1, ragged=None)
    x = synth.gen_layer(wl, 2)
    p = O.Params(**case.get("p", {}))
    rho = case.get("rho", wl.rho)
    _, host, _ = run_compress(wl, x, p, rho=rho)
    check_sequence(wl, x, host, 0, p, rho=rho)
    m = int(host["lengths"][0])
    if rho == 1.0:
        np.testing.assert_array_equal(host["kept_idx"][0, :m], np.arange(wl.n))
        np.testing.assert_array_equal(host["V_c"][0, :, :m], x["V"][0])
        np.testing.assert_array_equal(host["bias"][0, :, :m], 0.0)
    if p.alpha == 0.0:
        np.testing.assert_array_equal(host["bias"][0, :, :m], 0.0)


@pytest.mark.parametrize("per_head", [False, True])
def test_compress_exact_ties_take_the_lowest_positions(per_head):
    """Every token of a sequence identical: the attention of all fully visible candidates, and
    so their pooled scores, are exactly equal (bit-identical on the GPU as in the oracle), and
    the top-m_s is decided by the position tie-break alone: lower positions first.  The kept
    set must equal the oracle's exactly (no near-tie allowance)."""
    wl = SMALL["bf16_ragged"].with_(batch=2, ragged=None)
    x = synth.gen_layer(wl, 7)
    x["K"][:] = x["K"][:, :, :1, :]
    x["V"][:] = x["V"][:, :, :1, :]
    p = O.Params(select_mode=O.SELECT_PER_HEAD if per_head else O.SELECT_SHARED)
    _, host, _ = run_compress(wl, x, p)
    for b in range(wl.batch):
        n = int(x["n_len"][b])
        ref = O.compress(x["K"][b].astype(np.float64), x["V"][b].astype(np.float64),
                         x["Q_obs"][b].astype(np.float64), n, wl.rho, p)
        m = int(host["lengths"][b])
        assert m == ref.m
        if per_head:
            np.testing.assert_array_equal(host["kept_idx"][b, :, :m], ref.kept_idx)
        else:
            np.testing.assert_array_equal(host["kept_idx"][b, :m], ref.kept_idx)
            # the tie really decided it: the kept candidates are a prefix of the tied run
            kept = ref.kept_idx[ref.kept_idx < n - p.recent]
            assert kept[-1] < n - wl.obs_window


def test_compress_on_concurrent_streams_matches_one_stream():
    """Two layers compressed at once on two streams (a workspace each, as a caller compressing
    a model's layers after prefill would) give bitwise the outputs of compressing them one
    after the other on one stream."""
    wl = SMALL["bf16_ragged"]
    xs = [synth.gen_layer(wl, 20 + i) for i in range(2)]
    n_len = [int(v) for v in xs[0]["n_len"]]
    assert n_len == [int(v) for v in xs[1]["n_len"]]
    m_cap = api.capacity(max(n_len), wl.rho)
    shape = api.make_shape(wl.dtype, wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                           wl.obs_window, wl.n, m_cap)
    ins = [tuple(to_dev(x[k], wl.dtype) for k in ("K", "V", "Q_obs")) for x in xs]
    torch.cuda.synchronize()  # the inputs exist before any other stream reads them

    def run(streams):
        outs = []
        for i, st in enumerate(streams):
            with torch.cuda.stream(st):
                ws = api.Workspace(S.selkv_compress_workspace_size(shape), "cuda", st.cuda_stream)
                outs.append((api.compress(shape, n_len, wl.rho, *ins[i], debug=True, workspace=ws,
                                          stream=st.cuda_stream), ws))
        torch.cuda.synchronize()
        return outs

    side = [torch.cuda.Stream(), torch.cuda.Stream()]
    one = torch.cuda.Stream()
    par = run(side)
    seq = run([one, one])
    for (a, wa), (b, wb) in zip(par, seq):
        assert wa.errors() == 0 and wb.errors() == 0
        for name in ("K_c", "V_c", "bias", "lengths"):
            assert torch.equal(getattr(a, name), getattr(b, name)), name
        for name in ("kept_idx", "target", "gate", "ratio"):
            assert torch.equal(a.debug[name], b.debug[name]), name


def test_window_equals_sequence():
    wl = SMALL["tiny"].with_(n=96, obs_window=96, rho=0.5)
    x = synth.gen_layer(wl, 0)
    p = O.Params()
    _, host, _ = run_compress(wl, x, p)
    check_sequence(wl, x, host, 0, p)


def test_compress_parity_llama_layer():
    """One Llama-3-8B-shaped layer at 16k (32 q / 8 KV heads, d = 128, bf16, W = 64)."""
    wl = synth.WORKLOADS["llama_layer"]
    x = synth.gen_layer(wl, 0, threads=8)
    p = O.Params()
    _, host, _ = run_compress(wl, x, p)
    st = Stats()
    check_sequence(wl, x, host, 0, p, stats=st)
    print("llama_layer", dict(st))


def _decode_case(wl, layer, steps, use_bias=True, p=None):
    x = synth.gen_layer(wl, layer, threads=8)
    p = p or O.Params()
    per_head = p.select_mode == O.SELECT_PER_HEAD
    cache, host, _ = run_compress(wl, x, p, extra=steps)
    dec = synth.gen_decode(wl, layer, steps)
    Kc0 = cache.K_c.double().cpu().numpy()
    Vc0 = cache.V_c.double().cpu().numpy()
    bias0 = cache.bias.double().cpu().numpy()
    lens0 = cache.lengths.cpu().numpy().copy()
    ws = api.Workspace(S.selkv_decode_workspace_size(cache.shape))
    worst = (0.0, 0.0)
    for t in range(steps):
        q = to_dev(dec["q"][t], wl.dtype)
        kn, vn = to_dev(dec["k_new"][t], wl.dtype), to_dev(dec["v_new"][t], wl.dtype)
        out = api.decode(cache, q, kn, vn, use_bias=use_bias, workspace=ws).float().cpu().numpy()
        for b in range(wl.batch):
            L0 = int(lens0[b])
            Kc = np.concatenate([Kc0[b, :, :L0], dec["k_new"][:t + 1, b].transpose(1, 0, 2)], axis=1)
            Vc = np.concatenate([Vc0[b, :, :L0], dec["v_new"][:t + 1, b].transpose(1, 0, 2)], axis=1)
            if not use_bias:
                bs = None
            elif per_head:   # one bias row per KV head (Sec. 3.6, per-head mode)
                bs = np.concatenate([bias0[b, :, :L0], np.zeros((wl.num_kv_heads, t + 1))], axis=1)
            else:
                bs = np.concatenate([bias0[b, 0, :L0], np.zeros(t + 1)])
            want = O.decode(dec["q"][t, b], Kc, Vc, bs, L0 + t + 1)
            e = check_decode(out[b], want, wl.dtype, "step %d seq %d" % (t, b))
            worst = (max(worst[0], e[0]), max(worst[1], e[1]))
    torch.cuda.synchronize()
    assert ws.errors() == 0
    lens = cache.lengths.cpu().numpy()
    np.testing.assert_array_equal(lens, lens0 + steps)
    Kc = cache.K_c.float().cpu().numpy()
    Vc = cache.V_c.float().cpu().numpy()
    bias = cache.bias.cpu().numpy()
    for b in range(wl.batch):
        L0 = int(lens0[b])
        np.testing.assert_array_equal(Kc[b, :, L0:L0 + steps], dec["k_new"][:, b].transpose(1, 0, 2))
        np.testing.assert_array_equal(Vc[b, :, L0:L0 + steps], dec["v_new"][:, b].transpose(1, 0, 2))
        if use_bias:
            np.testing.assert_array_equal(bias[b, :, L0:L0 + steps], 0.0)
    return worst


@pytest.mark.parametrize("name", ["tiny", "bf16_ragged", "bf16_d64_g4", "fp32_d128", "bf16_g8_w64"])
def test_decode_parity_small(name):
    worst = _decode_case(SMALL[name], 0, steps=4)
    print(name, "decode worst max/mean abs", worst)


def test_decode_parity_tiny_16_steps():
    """The tiny workload's 16 decode steps with fresh N(0, 1) queries and appended rows."""
    worst = _decode_case(synth.WORKLOADS["tiny"], 0, steps=16)
    print("tiny 16 steps", worst)


def test_decode_parity_llama_layer():
    worst = _decode_case(synth.WORKLOADS["llama_layer"], 0, steps=3)
    print("llama_layer decode", worst)


def test_decode_without_bias_is_plain_attention():
    worst = _decode_case(SMALL["bf16_ragged"], 3, steps=2, use_bias=False)
    print("no bias", worst)


def test_decode_full_cache_uncompressed():
    """bias = NULL over an uncompressed cache (m_cap = n_cap, lengths = n): exact attention."""
    wl = SMALL["bf16_ragged"]
    x = synth.gen_layer(wl, 4)
    shape = api.make_shape(wl.dtype, wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                           wl.obs_window, wl.n, wl.n)
    cache = api.CompressedCache(shape=shape, K_c=to_dev(x["K"], wl.dtype), V_c=to_dev(x["V"], wl.dtype),
                                bias=torch.zeros((wl.batch, wl.num_kv_heads, wl.n), device="cuda"),
                                lengths=torch.from_numpy(x["n_len"].astype(np.int32)).cuda())
    dec = synth.gen_decode(wl, 4, 1)
    out = api.decode(cache, to_dev(dec["q"][0], wl.dtype), use_bias=False).float().cpu().numpy()
    for b in range(wl.batch):
        n = int(x["n_len"][b])
        want = O.decode(dec["q"][0, b], x["K"][b], x["V"][b], None, n)
        check_decode(out[b], want, wl.dtype)


def test_decode_edge_lengths():
    """Empty cache: without a new row out = 0; with one, out = v_new.  A full cache with an
    append sets the capacity flag and attends over the existing rows only."""
    wl = SMALL["tiny"]
    shape = api.make_shape("fp32", 2, 4, 2, 64, 32, 64, 64)
    cache = api.alloc_compressed(shape)
    g = torch.Generator().manual_seed(0)
    cache.K_c.copy_(torch.randn(cache.K_c.shape, generator=g))
    cache.V_c.copy_(torch.randn(cache.V_c.shape, generator=g))
    cache.lengths.copy_(torch.tensor([0, 64], dtype=torch.int32))
    q = torch.randn((2, 4, 64), generator=g).cuda()
    kn = torch.randn((2, 2, 64), generator=g).cuda()
    vn = torch.randn((2, 2, 64), generator=g).cuda()
    ws = api.Workspace(S.selkv_decode_workspace_size(shape))
    out = api.decode(cache, q, workspace=ws).cpu().numpy()
    np.testing.assert_array_equal(out[0], 0.0)
    assert ws.errors() == 0
    out = api.decode(cache, q, kn, vn, workspace=ws).cpu().numpy()
    for h in range(4):
        np.testing.assert_allclose(out[0, h], vn[0, h // 2].cpu().numpy(), rtol=1e-6)
    assert ws.errors() == S.SELKV_DEVERR_CAPACITY
    lens = cache.lengths.cpu().numpy()
    np.testing.assert_array_equal(lens, [1, 64])
    want = O.decode(q[1].cpu().double().numpy(), cache.K_c[1].cpu().double().numpy(),
                    cache.V_c[1].cpu().double().numpy(), cache.bias[1].cpu().double().numpy(), 64)
    check_decode(out[1], want, "fp32")


def test_decode_back_to_back_appends_sweep_the_split_slices():
    """bf16 decode calls enqueued back to back on one cache, each appending a row, while the
    lengths sweep through every point where the per-split row slices move.  Each launch reads
    the length before waiting for the previous launch (to prefetch and to issue its first tile
    early), so that read is often one row stale: both the kept and the discarded early first
    tile are exercised.  Every step must match exact attention over the rows present then
    (bias per row, 0 for appended rows)."""
    B, Hq, Hkv, d, m_cap = 2, 8, 2, 128, 4224
    L0 = [1, 700]
    T, burst = 3500, 25
    shape = api.make_shape("bf16", B, Hq, Hkv, d, 32, m_cap, m_cap)
    g = torch.Generator().manual_seed(21)
    cache = api.alloc_compressed(shape)
    cache.K_c.copy_(torch.randn(cache.K_c.shape, generator=g))
    cache.V_c.copy_(torch.randn(cache.V_c.shape, generator=g))
    cache.bias.copy_(0.5 * torch.rand(cache.bias.shape, generator=g))
    cache.lengths.copy_(torch.tensor(L0, dtype=torch.int32))
    qs = torch.randn((T, B, Hq, d), generator=g).to(torch.bfloat16).cuda()
    ks = torch.randn((T, B, Hkv, d), generator=g).to(torch.bfloat16).cuda()
    vs = torch.randn((T, B, Hkv, d), generator=g).to(torch.bfloat16).cuda()
    outs = torch.empty((burst, B, Hq, d), dtype=torch.bfloat16, device="cuda")
    Kh = cache.K_c.double().cpu().numpy()
    Vh = cache.V_c.double().cpu().numpy()
    bh = cache.bias.double().cpu().numpy()
    qh, kh, vh = (x.double().cpu().numpy() for x in (qs, ks, vs))
    ws = api.Workspace(S.selkv_decode_workspace_size(shape))
    for t0 in range(0, T, burst):
        for i in range(burst):
            t = t0 + i
            api.decode(cache, qs[t], ks[t], vs[t], out=outs[i], workspace=ws)
        got = outs.float().cpu().numpy()
        for i in range(burst):
            t = t0 + i
            for b in range(B):
                L = L0[b] + t
                Kh[b, :, L] = kh[t, b]
                Vh[b, :, L] = vh[t, b]
                bh[b, :, L] = 0.0
                want = O.decode(qh[t, b], Kh[b], Vh[b], bh[b], L + 1)
                check_decode(got[i, b], want, "bf16", "step %d seq %d" % (t, b))
    torch.cuda.synchronize()
    assert ws.errors() == 0
    np.testing.assert_array_equal(cache.lengths.cpu().numpy(), np.array(L0) + T)


@pytest.mark.parametrize("B,Hq,Hkv", [(48, 8, 4), (20, 128, 8)])
def test_decode_persistent_units_back_to_back(B, Hq, Hkv):
    """More (sequence, KV head) units than SMs, one split each (48 sequences x 4 KV heads, and
    20 x 8 with 16-head groups): the decode runs as persistent CTAs walking the units.  Ragged
    lengths with the edge cases of a 128-row tile and of the early loads (0, 1, 63-65, 127-129
    rows), 40 appending steps enqueued back to back in bursts; every sequence of every step
    against exact attention over its rows (bias per row, 0 for appended rows), then the lengths
    and the error word."""
    d, m_cap = 128, 600
    g = torch.Generator().manual_seed(33 + B)
    edge = [0, 1, 63, 64, 65, 127, 128, 129, 255, 256, 257, 511]
    L0 = (edge + [int(x) for x in torch.randint(0, 540, (max(0, B - len(edge)),), generator=g)])[:B]
    T, burst = 40, 10
    shape = api.make_shape("bf16", B, Hq, Hkv, d, 32, m_cap, m_cap)
    cache = api.alloc_compressed(shape)
    cache.K_c.copy_(torch.randn(cache.K_c.shape, generator=g))
    cache.V_c.copy_(torch.randn(cache.V_c.shape, generator=g))
    cache.bias.copy_(0.5 * torch.rand(cache.bias.shape, generator=g))
    cache.lengths.copy_(torch.tensor(L0, dtype=torch.int32))
    qs = torch.randn((T, B, Hq, d), generator=g).to(torch.bfloat16).cuda()
    ks = torch.randn((T, B, Hkv, d), generator=g).to(torch.bfloat16).cuda()
    vs = torch.randn((T, B, Hkv, d), generator=g).to(torch.bfloat16).cuda()
    outs = torch.empty((burst, B, Hq, d), dtype=torch.bfloat16, device="cuda")
    Kh = cache.K_c.double().cpu().numpy()
    Vh = cache.V_c.double().cpu().numpy()
    bh = cache.bias.double().cpu().numpy()
    qh, kh, vh = (x.double().cpu().numpy() for x in (qs, ks, vs))
    ws = api.Workspace(S.selkv_decode_workspace_size(shape))
    for t0 in range(0, T, burst):
        for i in range(burst):
            api.decode(cache, qs[t0 + i], ks[t0 + i], vs[t0 + i], out=outs[i], workspace=ws)
        got = outs.float().cpu().numpy()
        for i in range(burst):
            t = t0 + i
            for b in range(B):
                L = L0[b] + t
                Kh[b, :, L] = kh[t, b]
                Vh[b, :, L] = vh[t, b]
                bh[b, :, L] = 0.0
                want = O.decode(qh[t, b], Kh[b], Vh[b], bh[b], L + 1)
                check_decode(got[i, b], want, "bf16", "step %d seq %d" % (t, b))
    torch.cuda.synchronize()
    assert ws.errors() == 0
    np.testing.assert_array_equal(cache.lengths.cpu().numpy(), np.array(L0) + T)


def test_repeat_runs_are_bitwise_identical():
    wl = SMALL["bf16_ragged"]
    x = synth.gen_layer(wl, 5)
    p = O.Params()
    _, h1, _ = run_compress(wl, x, p)
    _, h2, _ = run_compress(wl, x, p)
    for k in ("attn", "score", "kept_idx", "target", "gate", "V_c", "bias"):
        np.testing.assert_array_equal(h1[k], h2[k], err_msg=k)


# ---------------------------------------------------------------- per-head selection mode
PER_HEAD = {
    "tiny": SMALL["tiny"],                                          # fp32, G = 2
    "bf16_mha": synth.WORKLOADS["llama_layer"].with_(name="bf16_mha", batch=2, n=2600,
                                                     num_q_heads=4, num_kv_heads=4,
                                                     ragged=(0.6, 1.0), seed=21),   # G = 1
    "bf16_ragged": SMALL["bf16_ragged"],                            # bf16, G = 4
}


@pytest.mark.parametrize("name", list(PER_HEAD))
def test_compress_parity_per_head(name):
    """Sec. 3.3 per-head selection and Sec. 3.6 per-head bias against the oracle."""
    wl = PER_HEAD[name]
    x = synth.gen_layer(wl, 0)
    p = O.Params(select_mode=O.SELECT_PER_HEAD)
    _, host, _ = run_compress(wl, x, p)
    st = Stats()
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p, stats=st)
    print(name, dict(st))


def test_per_head_gate_closed_is_eviction():
    wl = PER_HEAD["bf16_mha"]
    x = synth.gen_layer(wl, 1)
    p = O.Params(select_mode=O.SELECT_PER_HEAD, gate_mode=O.GATE_CLOSED)
    _, host, _ = run_compress(wl, x, p)
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p)
        m = int(host["lengths"][b])
        for kv in range(wl.num_kv_heads):
            kept = host["kept_idx"][b, kv, :m]
            np.testing.assert_array_equal(host["V_c"][b, kv, :m], x["V"][b, kv][kept])
        np.testing.assert_array_equal(host["bias"][b, :, :m], 0.0)


def test_per_head_with_one_kv_head_matches_shared():
    """One KV head: both selection modes give the same cache, bias and targets on the GPU."""
    wl = SMALL["bf16_ragged"].with_(num_q_heads=4, num_kv_heads=1, batch=2, seed=22)
    x = synth.gen_layer(wl, 0)
    _, h_sh, _ = run_compress(wl, x, O.Params())
    _, h_ph, _ = run_compress(wl, x, O.Params(select_mode=O.SELECT_PER_HEAD))
    for b in range(wl.batch):
        m = int(h_sh["lengths"][b])
        n = int(x["n_len"][b])
        np.testing.assert_array_equal(h_ph["kept_idx"][b, 0, :m], h_sh["kept_idx"][b, :m])
        for k in ("K_c", "V_c", "bias", "ratio"):
            np.testing.assert_array_equal(h_ph[k][b, :, :m], h_sh[k][b, :, :m])
        np.testing.assert_array_equal(h_ph["target"][b, :, :n], h_sh["target"][b, :, :n])


@pytest.mark.parametrize("name", ["tiny", "bf16_mha"])
def test_decode_parity_per_head(name):
    """Decode over per-head caches: each KV head's own rows and bias row."""
    worst = _decode_case(PER_HEAD[name], 0, steps=3, p=O.Params(select_mode=O.SELECT_PER_HEAD))
    print(name, "per-head decode worst max/mean abs", worst)


# ---------------------------------------------------------------- Eq. 7: RoPE repositioning
@pytest.mark.parametrize("name,layout,mode", [
    ("tiny", O.ROPE_HALF, O.SELECT_SHARED),
    ("bf16_ragged", O.ROPE_HALF, O.SELECT_SHARED),
    ("bf16_d64_g4", O.ROPE_INTERLEAVED, O.SELECT_SHARED),
    ("fp32_d128", O.ROPE_INTERLEAVED, O.SELECT_SHARED),
])
def test_compress_rope_reposition(name, layout, mode):
    wl = SMALL[name]
    x = synth.gen_layer(wl, 3)
    p = O.Params(rope=layout, rope_theta=10000.0, select_mode=mode)
    _, host, _ = run_compress(wl, x, p)
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p)


def test_compress_rope_reposition_per_head_large_base():
    wl = PER_HEAD["bf16_mha"]
    x = synth.gen_layer(wl, 4)
    p = O.Params(rope=O.ROPE_HALF, rope_theta=500000.0, select_mode=O.SELECT_PER_HEAD)
    _, host, _ = run_compress(wl, x, p)
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p)


# ---------------------------------------------------------------- count bias (KeepKV variant)
@pytest.mark.parametrize("name,mode,alpha", [
    ("bf16_ragged", O.SELECT_SHARED, 1.0),
    ("tiny", O.SELECT_SHARED, 0.5),
    ("bf16_mha", O.SELECT_PER_HEAD, 1.0),
])
def test_compress_count_bias(name, mode, alpha):
    wl = SMALL.get(name) or PER_HEAD[name]
    x = synth.gen_layer(wl, 5)
    p = O.Params(bias_mode=O.BIAS_COUNT, select_mode=mode, alpha=alpha)
    _, host, _ = run_compress(wl, x, p)
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p)


# ---------------------------------------------------------------- full cosine routing (Sec. 3.4)
@pytest.mark.parametrize("name,mode", [
    ("tiny", O.SELECT_SHARED),
    ("bf16_ragged", O.SELECT_SHARED),
    ("bf16_d64_g4", O.SELECT_SHARED),
    ("fp32_d128", O.SELECT_SHARED),
    ("bf16_mha", O.SELECT_PER_HEAD),
])
def test_compress_cosine_routing(name, mode):
    wl = SMALL.get(name) or PER_HEAD[name]
    x = synth.gen_layer(wl, 6)
    p = O.Params(routing=O.ROUTE_COSINE, select_mode=mode)
    _, host, _ = run_compress(wl, x, p)
    st = Stats()
    for b in range(wl.batch):
        check_sequence(wl, x, host, b, p, stats=st)
    print(name, dict(st))


@pytest.mark.parametrize("case", [
    dict(p=dict(gate_mode=O.GATE_OPEN)),
    dict(p=dict(gate_mode=O.GATE_CLOSED)),
    dict(p=dict(bias_mode=O.BIAS_COUNT, alpha=1.0)),
    dict(rho=1.0),                                   # nothing evicted
    dict(rho=16 / 3001 + 1e-9),                      # only the recent window is kept
    dict(rho=0.9),                                   # several 256-slot tiles and a ragged one
])
def test_compress_cosine_routing_cases(case):
    wl = SMALL["bf16_ragged"].with_(batch=1, ragged=None)
    x = synth.gen_layer(wl, 7)
    p = O.Params(routing=O.ROUTE_COSINE, **case.get("p", {}))
    rho = case.get("rho", wl.rho)
    _, host, _ = run_compress(wl, x, p, rho=rho)
    check_sequence(wl, x, host, 0, p, rho=rho)


def test_cosine_routing_repeat_is_bitwise_identical():
    wl = SMALL["bf16_ragged"]
    x = synth.gen_layer(wl, 8)
    p = O.Params(routing=O.ROUTE_COSINE)
    _, h1, _ = run_compress(wl, x, p)
    _, h2, _ = run_compress(wl, x, p)
    for k in ("target", "gate", "V_c", "ratio", "bias"):
        np.testing.assert_array_equal(h1[k], h2[k], err_msg=k)


def test_cosine_routing_hub_and_zero_rows():
    """Adversarial values: many evicted rows parallel to one kept row (a hub slot with hundreds
    of contributors), zero value rows, and exact ties between kept rows."""
    wl = SMALL["bf16_ragged"].with_(batch=1, ragged=None, seed=31)
    x = synth.gen_layer(wl, 0)
    V = x["V"]
    V0 = V[0]                                   # [Hkv][n_cap][d], a view
    r = np.random.default_rng(5)
    n = wl.n
    hub = r.choice(n, 700, replace=False)
    # powers of two keep the copies exact in bf16
    V0[:, hub] = V0[:, hub[:1]] * r.choice([0.5, 1.0, 2.0], size=(1, 700, 1)).astype(V.dtype)
    V0[:, r.choice(n, 40, replace=False)] = 0
    twins = r.choice(n, 60, replace=False)
    V0[:, twins[30:]] = V0[:, twins[:30]]
    x["V"] = V
    p = O.Params(routing=O.ROUTE_COSINE)
    _, host, _ = run_compress(wl, x, p)
    st = Stats()
    check_sequence(wl, x, host, 0, p, stats=st)
    print(dict(st))


# ---------------------------------------------------------------- compensation averaged across layers
@pytest.mark.parametrize("name,mode,bias_mode,alpha", [
    ("bf16_ragged", O.SELECT_SHARED, O.BIAS_RATIO, 0.5),
    ("tiny", O.SELECT_SHARED, O.BIAS_COUNT, 1.0),
    ("bf16_mha", O.SELECT_PER_HEAD, O.BIAS_RATIO, 0.5),
    ("bf16_d64_g4", O.SELECT_SHARED, O.BIAS_RATIO, 0.0),
])
def test_layer_average_bias(name, mode, bias_mode, alpha):
    """Three layers compressed on the GPU (each checked against the oracle), then the biases
    replaced by their cross-layer average (R21) through the C ABI, against the oracle's average
    of the oracle's per-layer values."""
    wl = SMALL.get(name) or PER_HEAD[name]
    p = O.Params(select_mode=mode, bias_mode=bias_mode, alpha=alpha)
    L = 3
    caches, refs = [], []
    for layer in range(L):
        x = synth.gen_layer(wl, layer)
        cache, host, _ = run_compress(wl, x, p)
        caches.append(cache)
        refs.append([check_sequence(wl, x, host, b, p) for b in range(wl.batch)])
    shape = caches[0].shape
    ws = api.Workspace(S.selkv_layer_average_workspace_size(shape))
    S.check(S.selkv_layer_average_bias(shape, params_of(p), [c.debug["kept_idx"] for c in caches],
                                       [c.bias for c in caches], caches[0].lengths, ws.buf, ws.nbytes),
            "selkv_layer_average_bias")
    torch.cuda.synchronize()
    assert ws.errors() == 0
    count = bias_mode == O.BIAS_COUNT
    for b in range(wl.batch):
        m, n = refs[0][b]["m"], refs[0][b]["n"]
        if alpha == 0.0:
            for c in caches:
                np.testing.assert_array_equal(c.bias[b, :, :m].cpu().numpy(), 0.0)
            continue
        # the oracle's per-slot quantity of each layer: R (ratio bias) or M (count bias)
        x_l = [np.expm1(r[b]["bias"] / alpha) for r in refs]
        q_l = [x if count else 1.0 + x for x in x_l]
        want = O.layer_average_bias(q_l, [r[b]["kept_idx"] for r in refs], n, alpha, count)
        for layer in range(L):
            got = caches[layer].bias[b, :, :m].cpu().numpy().astype(np.float64)
            exp = want[layer] if mode == O.SELECT_PER_HEAD else np.broadcast_to(want[layer], got.shape)
            err = np.abs(got - exp).max()
            assert err <= BIAS_ATOL, "layer %d seq %d: bias err %.3g" % (layer, b, err)


def test_layer_average_one_layer_is_identity():
    wl = SMALL["bf16_ragged"]
    x = synth.gen_layer(wl, 0)
    p = O.Params()
    cache, host, _ = run_compress(wl, x, p)
    before = cache.bias.clone()
    ws = api.Workspace(S.selkv_layer_average_workspace_size(cache.shape))
    S.check(S.selkv_layer_average_bias(cache.shape, params_of(p), [cache.debug["kept_idx"]], [cache.bias],
                                       cache.lengths, ws.buf, ws.nbytes), "selkv_layer_average_bias")
    torch.cuda.synchronize()
    for b in range(wl.batch):
        m = int(host["lengths"][b])
        np.testing.assert_allclose(cache.bias[b, :, :m].cpu().numpy(), before[b, :, :m].cpu().numpy(),
                                   rtol=0, atol=2e-6)


# ---------------------------------------------------------------- scoring stage on its own
@pytest.mark.parametrize("name", ["tiny", "bf16_ragged", "bf16_d64_g4", "bf16_g8_w64", "bf16_g16_w24_d64"])
def test_score_entry_point(name):
    """selkv_score (Sec. 3.1 re-pass, Eq. 1's attention sums): a within ATTN_RTOL of the
    oracle; bitwise the `attn` of selkv_compress; the two passes run as separate calls
    (row statistics, then column sums) give bitwise the one-call result."""
    from parity import ATTN_RTOL
    wl = SMALL[name]
    x = synth.gen_layer(wl, 9)
    n_len = [int(v) for v in x["n_len"]]
    m_cap = api.capacity(max(n_len), wl.rho)
    shape = api.make_shape(wl.dtype, wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                           wl.obs_window, wl.n, m_cap)
    K, Q = to_dev(x["K"], wl.dtype), to_dev(x["Q_obs"], wl.dtype)
    ws = api.Workspace(S.selkv_score_workspace_size(shape))
    a_all = torch.full((wl.batch, wl.num_kv_heads, wl.n), -1.0, device="cuda")
    a_two = torch.full_like(a_all, -2.0)
    S.check(S.selkv_score(shape, n_len, K, Q, a_all, S.SELKV_SCORE_ALL, ws.buf, ws.nbytes), "score")
    S.check(S.selkv_score(shape, n_len, K, Q, None, S.SELKV_SCORE_ROWSTATS, ws.buf, ws.nbytes), "rowstats")
    S.check(S.selkv_score(shape, n_len, K, Q, a_two, S.SELKV_SCORE_COLSUMS, ws.buf, ws.nbytes), "colsums")
    torch.cuda.synchronize()
    assert ws.errors() == 0
    _, host, _ = run_compress(wl, x, O.Params())
    got, two = a_all.cpu().numpy(), a_two.cpu().numpy()
    for b in range(wl.batch):
        n = n_len[b]
        want = O.cumulative_attention(x["Q_obs"][b].astype(np.float64), x["K"][b].astype(np.float64), n)
        err = np.abs(got[b, :, :n] - want) / (np.abs(want) + 1e-30)
        assert err.max() <= ATTN_RTOL, "attention rel err %.3g" % err.max()
        np.testing.assert_array_equal(got[b, :, :n], host["attn"][b, :, :n])
        np.testing.assert_array_equal(two[b, :, :n], got[b, :, :n])
        assert (got[b, :, n:] == -1.0).all(), "entries past n_b were written"


def test_decode_after_a_kernel_that_rewrites_the_lengths():
    """The decode starts on its slice before the kernel enqueued just before it has finished,
    planning from a length it reads without ordering.  Here that previous kernel rewrites the
    lengths (a torch fill on the same stream: shorter, then longer than the decode before it
    left them), so the early plan is stale: every output must still equal exact attention over
    the rows the new length names."""
    B, Hq, Hkv, d, m_cap = 2, 8, 2, 128, 4096
    shape = api.make_shape("bf16", B, Hq, Hkv, d, 32, m_cap, m_cap)
    g = torch.Generator().manual_seed(5)
    cache = api.alloc_compressed(shape)
    cache.K_c.copy_(torch.randn(cache.K_c.shape, generator=g))
    cache.V_c.copy_(torch.randn(cache.V_c.shape, generator=g))
    cache.bias.copy_(0.3 * torch.rand(cache.bias.shape, generator=g))
    ws = api.Workspace(S.selkv_decode_workspace_size(shape))
    Kh = cache.K_c.double().cpu().numpy()
    Vh = cache.V_c.double().cpu().numpy()
    bh = cache.bias.double().cpu().numpy()
    for L in (3000, 1100, 3900, 700, 2600):
        cache.lengths.fill_(L)   # a kernel on the current stream, right before the decode
        q = torch.randn((B, Hq, d), generator=g).to(torch.bfloat16).cuda()
        out = api.decode(cache, q, workspace=ws).float().cpu().numpy()
        qh = q.double().cpu().numpy()
        for b in range(B):
            want = O.decode(qh[b], Kh[b], Vh[b], bh[b], L)
            check_decode(out[b], want, "bf16", "length %d seq %d" % (L, b))
    torch.cuda.synchronize()
    assert ws.errors() == 0


def test_compress_and_decode_at_the_maximum_batch():
    """SELKV_MAX_BATCH sequences of a few hundred tokens each (ragged, the smallest near the
    window): every sequence passes the structural checks, eight spread over the batch are
    checked against the oracle stage by stage, and one decode step of all of them against
    exact attention over each one's compressed rows."""
    from parity import check_properties
    wl = synth.WORKLOADS["llama_layer"].with_(name="max_batch", batch=S.SELKV_MAX_BATCH, n=320,
                                              num_q_heads=8, num_kv_heads=2, obs_window=24,
                                              ragged=(0.3, 1.0), seed=17)
    x = synth.gen_layer(wl, 0, threads=16)
    p = O.Params()
    cache, host, _ = run_compress(wl, x, p, extra=1)
    check_properties(wl, x, host, p)
    for b in np.linspace(0, wl.batch - 1, 8).astype(int):
        check_sequence(wl, x, host, int(b), p)
    dec = synth.gen_decode(wl, 0, 1)
    Kc = cache.K_c.double().cpu().numpy()
    Vc = cache.V_c.double().cpu().numpy()
    bias = cache.bias.double().cpu().numpy()
    lens = cache.lengths.cpu().numpy().copy()
    ws = api.Workspace(S.selkv_decode_workspace_size(cache.shape))
    out = api.decode(cache, to_dev(dec["q"][0], wl.dtype), to_dev(dec["k_new"][0], wl.dtype),
                     to_dev(dec["v_new"][0], wl.dtype), workspace=ws).float().cpu().numpy()
    torch.cuda.synchronize()
    assert ws.errors() == 0
    np.testing.assert_array_equal(cache.lengths.cpu().numpy(), lens + 1)
    for b in range(0, wl.batch, 37):
        L = int(lens[b])
        K1 = np.concatenate([Kc[b, :, :L], dec["k_new"][0, b][:, None]], axis=1)
        V1 = np.concatenate([Vc[b, :, :L], dec["v_new"][0, b][:, None]], axis=1)
        b1 = np.concatenate([bias[b, 0, :L], [0.0]])
        check_decode(out[b], O.decode(dec["q"][0, b], K1, V1, b1, L + 1), wl.dtype, "seq %d" % b)
