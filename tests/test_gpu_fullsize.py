"""GPU parity at the workloads' full sizes, in the launch configuration bench.py times.

The oracle checks sampled sequences stage by stage (the same rules as the small parity tests);
every sequence of every compressed layer also passes the structural checks of
parity.check_properties; decode is compared with the oracle's decode over the GPU's own
compressed cache for sampled sequences."""
import numpy as np
import pytest
import torch

import synth
from oracle import selkv_oracle as O
from paper_2607_16213_gb300 import api
import paper_2607_16213_gb300 as S

from parity import Stats, check_decode, check_keys, check_properties, check_sequence, run_compress, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16213_gb300 import build as b
    b.build()
    S.library()


def _decode_sampled(wl, cache, layer, seqs, steps=2, per_head=False):
    """Decode `steps` tokens (appending) and compare sampled sequences with the oracle's decode
    over the GPU's compressed cache as it stood before each step."""
    dec = synth.gen_decode(wl, layer, steps)
    ws = api.Workspace(S.selkv_decode_workspace_size(cache.shape))
    for t in range(steps):
        Kc = cache.K_c.double().cpu().numpy()
        Vc = cache.V_c.double().cpu().numpy()
        bias = cache.bias.double().cpu().numpy()
        lens = cache.lengths.cpu().numpy().copy()
        out = api.decode(cache, to_dev(dec["q"][t], wl.dtype), to_dev(dec["k_new"][t], wl.dtype),
                         to_dev(dec["v_new"][t], wl.dtype), workspace=ws).float().cpu().numpy()
        for b in seqs:
            L = int(lens[b])
            K1 = np.concatenate([Kc[b, :, :L], dec["k_new"][t, b][:, None]], axis=1)
            V1 = np.concatenate([Vc[b, :, :L], dec["v_new"][t, b][:, None]], axis=1)
            if per_head:   # one bias row per KV head
                b1 = np.concatenate([bias[b, :, :L], np.zeros((wl.num_kv_heads, 1))], axis=1)
            else:
                b1 = np.concatenate([bias[b, 0, :L], [0.0]])
            want = O.decode(dec["q"][t, b], K1, V1, b1, L + 1)
            check_decode(out[b], want, wl.dtype, "layer %d step %d seq %d" % (layer, t, b))
    torch.cuda.synchronize()
    assert ws.errors() == 0


def test_long_100k_layer():
    """One layer of the 100k-context workload: full stage-by-stage parity and decode."""
    wl = synth.WORKLOADS["long_100k"]
    x = synth.gen_layer(wl, 7, threads=16)
    p = O.Params()
    cache, host, _ = run_compress(wl, x, p, extra=wl.decode_steps + 1)
    st = Stats()
    check_sequence(wl, x, host, 0, p, stats=st)
    check_properties(wl, x, host, p)
    print("long_100k", dict(st))
    _decode_sampled(wl, cache, 7, [0], steps=2)


@pytest.mark.parametrize("layer,seq", [(0, 0), (31, 3)])
def test_llama_32l_b4_layers(layer, seq):
    """Layers of the 32-layer, batch-4, 32k workload: one sequence against the oracle, all
    sequences against the structural checks, decode on two sequences."""
    wl = synth.WORKLOADS["llama_32l_b4"]
    x = synth.gen_layer(wl, layer, threads=16)
    p = O.Params()
    cache, host, _ = run_compress(wl, x, p, extra=wl.decode_steps + 1)
    st = Stats()
    check_sequence(wl, x, host, seq, p, stats=st)
    check_properties(wl, x, host, p)
    print("llama_32l_b4 layer", layer, dict(st))
    _decode_sampled(wl, cache, layer, [seq, (seq + 1) % wl.batch], steps=2)


SWEEP = [(1, 8192, 0.10), (8, 8192, 0.50), (64, 8192, 0.25), (64, 8192, 0.50), (8, 32768, 0.25),
         (32, 8192, 0.10), (1, 131072, 0.25), (1, 32768, 0.50)]


@pytest.mark.parametrize("batch,n,rho", SWEEP)
def test_serving_sweep_point(batch, n, rho):
    """Points of the batched serving sweep (ragged lengths): the shortest and the longest
    sequence against the oracle, every sequence against the structural checks, decode on the
    same two."""
    wl = synth.sweep(batch, n, rho)
    x = synth.gen_layer(wl, 0, threads=16)
    p = O.Params()
    cache, host, _ = run_compress(wl, x, p, extra=wl.decode_steps + 1)
    lens = x["n_len"]
    picks = sorted({int(np.argmin(lens)), int(np.argmax(lens))})
    st = Stats()
    for b in picks:
        check_sequence(wl, x, host, b, p, stats=st)
    check_properties(wl, x, host, p)
    print(wl.name, dict(st))
    _decode_sampled(wl, cache, 0, picks, steps=2)


def test_longchat_mha_layer_per_head():
    """One layer of the MHA workload (32 query heads = 32 KV heads, n = 31,500) in the per-head
    selection mode: stage-by-stage parity of every head, decode with per-head bias rows."""
    wl = synth.WORKLOADS["longchat_mha_31k"]
    x = synth.gen_layer(wl, 5, threads=16)
    p = O.Params(select_mode=O.SELECT_PER_HEAD)
    cache, host, _ = run_compress(wl, x, p, extra=wl.decode_steps + 1)
    st = Stats()
    check_sequence(wl, x, host, 0, p, stats=st)
    print("longchat_mha_31k per-head", dict(st))
    _decode_sampled(wl, cache, 5, [0], steps=2, per_head=True)


def test_long_100k_layer_rope_shifts():
    """RoPE repositioning at 100k context (shifts up to ~75,000 positions, base 500,000): every
    KV head's repositioned keys against the oracle's Eq. 7."""
    wl = synth.WORKLOADS["long_100k"]
    x = synth.gen_layer(wl, 9, threads=16)
    p = O.Params(rope=O.ROPE_HALF, rope_theta=500000.0)
    _, host, _ = run_compress(wl, x, p)
    m = int(host["lengths"][0])
    kept = host["kept_idx"][0, :m].astype(np.int64)
    assert kept[-1] - (m - 1) > 50000
    for kv in range(wl.num_kv_heads):
        check_keys(host["K_c"][0, kv, :m], x["K"][0, kv][kept].astype(np.float64), kept, p, wl.dtype)


def test_llama70b_layer_wide_group():
    """One layer of the G = 8 workload (64 query heads over 8 KV heads, 16k, W = 64: G W = 512
    window rows per KV head, scored on the tensor cores in two row halves): stage-by-stage
    parity and decode."""
    wl = synth.WORKLOADS["llama70b_layer"]
    x = synth.gen_layer(wl, 0, threads=16)
    p = O.Params()
    cache, host, _ = run_compress(wl, x, p, extra=3)
    st = Stats()
    check_sequence(wl, x, host, 0, p, stats=st)
    check_properties(wl, x, host, p)
    _decode_sampled(wl, cache, 0, [0], steps=2)
