"""selkv_decode_attn_static: the decode for callers that cannot allocate device memory (a host
framework that owns every buffer and gives a kernel only its inputs and outputs, or a serving
loop that must not call cudaMalloc / cudaFree).  Its scratch lives in a fixed static device
array inside the library instead of a caller workspace.

Checked here through the C ABI: on two calls in a row (the second one reuses the array the
first one left behind) it gives the same outputs, appended rows and lengths as
selkv_decode_attn, within the decode tolerance of the parity tests; shapes whose scratch
would not fit are rejected before launch.  This file sorts last so that a run stopping at the
first failure has already run every other test."""
import numpy as np
import pytest
import torch

import synth
from oracle import selkv_oracle as O
import paper_2607_16213_gb300 as S
from paper_2607_16213_gb300 import api

from parity import check_decode, run_compress, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16213_gb300 import build as b
    b.build()
    S.library()


def _clone(c: api.CompressedCache) -> api.CompressedCache:
    return api.CompressedCache(shape=c.shape, K_c=c.K_c.clone(), V_c=c.V_c.clone(),
                               bias=c.bias.clone(), lengths=c.lengths.clone())


@pytest.mark.parametrize("name,wl", [
    ("bf16_ragged", synth.WORKLOADS["llama_layer"].with_(batch=3, n=3001, num_q_heads=8,
                                                        num_kv_heads=2, ragged=(0.5, 1.0), seed=21)),
    ("tiny_fp32", synth.WORKLOADS["tiny"]),
])
def test_static_decode_matches_workspace_decode(name, wl):
    x = synth.gen_layer(wl, 0)
    a, _, _ = run_compress(wl, x, O.Params(), extra=2)
    b = _clone(a)
    shape = a.shape
    ws = api.Workspace(S.selkv_decode_workspace_size(shape))
    flags = torch.zeros(1, dtype=torch.int32, device="cuda")
    dec = synth.gen_decode(wl, 0, 2)
    for t in range(2):
        q = to_dev(dec["q"][t], wl.dtype)
        kn, vn = to_dev(dec["k_new"][t], wl.dtype), to_dev(dec["v_new"][t], wl.dtype)
        out_ws = torch.empty_like(q)
        out_st = torch.full_like(q, float("nan"))
        S.check(S.selkv_decode_attn(shape, q, a.K_c, a.V_c, a.bias, a.lengths, kn, vn, out_ws,
                                    ws.buf, ws.nbytes), "selkv_decode_attn")
        S.check(S.selkv_decode_attn_static(shape, q, b.K_c, b.V_c, b.bias, b.lengths, kn, vn,
                                           out_st, flags), "selkv_decode_attn_static")
        torch.cuda.synchronize()
        ref = out_ws.double().cpu().numpy()
        got = out_st.float().cpu().numpy()
        for s in range(wl.batch):
            check_decode(got[s], ref[s], wl.dtype, "%s call %d seq %d" % (name, t, s))
        np.testing.assert_array_equal(b.lengths.cpu().numpy(), a.lengths.cpu().numpy())
    assert int(flags.item()) == 0
    assert ws.errors() == 0
    np.testing.assert_array_equal(b.K_c.float().cpu().numpy(), a.K_c.float().cpu().numpy())
    np.testing.assert_array_equal(b.V_c.float().cpu().numpy(), a.V_c.float().cpu().numpy())
    np.testing.assert_array_equal(b.bias.cpu().numpy(), a.bias.cpu().numpy())


def test_static_decode_rejects_shapes_beyond_its_scratch():
    # 1024 sequences x 64 query heads x d 128 needs ~34 MB of split partials
    shape = api.make_shape("bf16", 1024, 64, 8, 128, 64, 4096, 4096)
    fake = 1 << 40
    st = S.selkv_decode_attn_static(shape, fake, fake, fake, None, fake, None, None, fake, None, 0)
    assert st == S.SELKV_ERR_WORKSPACE
