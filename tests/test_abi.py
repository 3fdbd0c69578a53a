"""The C-ABI library on the host: it loads, exports every function include/selkv.h declares,
sizes workspaces, and rejects invalid arguments with a status code before any CUDA call (so
these run without a GPU; no call here reaches a kernel launch)."""
import os
import subprocess

import pytest

import paper_2607_16213_gb300 as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FAKE = 1 << 40          # a 256-aligned address that is never dereferenced: every call below
                        # fails validation first


@pytest.fixture(scope="module")
def lib():
    from paper_2607_16213_gb300 import build as b
    b.build()
    return S.library()


def shape(**kw):
    base = dict(dtype=S.SELKV_BF16, batch=1, num_q_heads=32, num_kv_heads=8, head_dim=128,
                obs_window=64, n_cap=16384, m_cap=4160)
    base.update(kw)
    return S.selkv_shape(**base)


def test_exports_every_declared_symbol(lib):
    names = S.exported_symbols()
    assert {"selkv_compress", "selkv_decode_attn", "selkv_compress_workspace_size",
            "selkv_decode_workspace_size", "selkv_workspace_init", "selkv_workspace_error",
            "selkv_status_string", "selkv_kernel_launches"} <= set(names)
    out = subprocess.run(["nm", "-D", "--defined-only", S.library_path()], capture_output=True,
                         text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    for n in names:
        assert n in exported, n
        assert hasattr(lib, n)
    assert all(e.startswith("selkv_") for e in exported), exported


def test_status_strings(lib):
    assert S.selkv_status_string(S.SELKV_OK) == "ok"
    assert "workspace" in S.selkv_status_string(S.SELKV_ERR_WORKSPACE)
    assert S.selkv_status_string(99) == "unknown status"


def test_last_cuda_error_starts_clear(lib):
    # nothing has failed on this thread: cudaSuccess, by its runtime name
    code, name = S.selkv_last_cuda_error()
    assert code == 0 and name == "cudaSuccess"


def test_workspace_sizes(lib):
    s = shape()
    c = S.selkv_compress_workspace_size(s)
    d = S.selkv_decode_workspace_size(s)
    assert c > 256 and d > 256 and c % 256 == 0 and d % 256 == 0
    assert S.selkv_compress_workspace_size(shape(n_cap=32768)) > c
    assert S.selkv_compress_workspace_size(shape(num_kv_heads=7)) == 0      # 32 % 7 != 0
    assert S.selkv_compress_workspace_size(shape(batch=0)) == 0
    assert S.selkv_decode_workspace_size(shape(dtype=5)) == 0


def _decode_splits(s) -> int:
    """The split count the host planned for a decode shape, read back from the decode
    workspace size: a 256-byte header, the per-(b, kv) and per-b arrival counters, and one
    record per (b, kv) of G S d partial outputs plus G S (max, sum) pairs padded to 16 bytes,
    each region rounded up to 256 bytes."""
    r256 = lambda x: (x + 255) // 256 * 256
    G, units = s.num_q_heads // s.num_kv_heads, s.batch * s.num_kv_heads
    total = S.selkv_decode_workspace_size(s)
    for splits in range(1, 65):
        rec = G * splits * s.head_dim + (G * splits * 2 + 3) // 4 * 4
        if 256 + r256(units * 4) + r256(s.batch * 4) + r256(units * rec * 4) == total:
            return splits
    raise AssertionError("no split count gives %d bytes" % total)


@pytest.mark.parametrize("batch,m_cap,splits", [
    (1, 25280, 19),    # 100k context, 25% kept: one wave of 8 x 19 CTAs
    (4, 8512, 4),      # batch 4 x 32k at 25%: 4 splits in one wave, not 9 in two
    (1, 512, 8),       # short cache: splits with a combine beat one CTA streaming alone
    (32, 8128, 4),     # 256 units (under three waves): the units keep their splits
    (64, 2048, 1),     # 512 short units: one split each (the persistent walk)
    (64, 4096, 1),     # 512 units of at most 8192 rows: one split, waves counted fractionally
    (64, 16256, 2),    # longer units keep their splits
])
def test_decode_split_plan(lib, batch, m_cap, splits):
    """The split model's choices for the workloads it was tuned on (bf16, 32 query / 8 KV
    heads, d = 128), as the workspace size shows them."""
    assert _decode_splits(shape(batch=batch, m_cap=m_cap)) == splits


def _compress(s, n_len, rho=0.25, params=None, ptrs=None, ws=FAKE, wsb=1 << 40):
    p = params or S.selkv_params.defaults()
    t = dict(K=FAKE, V=FAKE, Q=FAKE, Kc=FAKE, Vc=FAKE, bias=FAKE, lengths=FAKE)
    t.update(ptrs or {})
    return S.selkv_compress(s, n_len, rho, p, t["K"], t["V"], t["Q"], t["Kc"], t["Vc"], t["bias"],
                            t["lengths"], None, ws, wsb, 0)


@pytest.mark.parametrize("case", [
    dict(n_len=[16384], rho=0.0),                 # rho must be in (0, 1]
    dict(n_len=[16384], rho=1.5),
    dict(n_len=[40]),                              # W = 64 > n_b
    dict(n_len=[20000]),                           # n_b > n_cap
    dict(n_len=[100], rho=0.1),                    # m = 10 < recent window 16
    dict(n_len=[16384], rho=0.5),                  # m = 8192 > m_cap
    dict(n_len=[16384], ptrs=dict(K=0)),           # NULL tensor
    dict(n_len=[16384], ptrs=dict(V=FAKE + 8)),    # misaligned tensor
    dict(n_len=[16384], params=S.selkv_params.defaults(pool_kernel=4)),   # even kernel
    dict(n_len=[16384], params=S.selkv_params.defaults(gate_mode=7)),
    dict(n_len=[16384], params=S.selkv_params.defaults(alpha=float("nan"))),
])
def test_compress_rejects_invalid_arguments(lib, case):
    assert _compress(shape(), **case) == S.SELKV_ERR_INVALID_ARG


def test_compress_unsupported_and_workspace(lib):
    assert _compress(shape(head_dim=96), [16384]) == S.SELKV_ERR_UNSUPPORTED
    assert _compress(shape(), [16384], params=S.selkv_params.defaults(bucket=64)) == S.SELKV_ERR_UNSUPPORTED
    assert _compress(shape(), [16384], ws=0) == S.SELKV_ERR_WORKSPACE
    assert _compress(shape(), [16384], ws=FAKE + 16) == S.SELKV_ERR_WORKSPACE
    assert _compress(shape(), [16384], wsb=1024) == S.SELKV_ERR_WORKSPACE
    assert _compress(shape(batch=2), [16384, 16384], ptrs=dict(Q=None)) == S.SELKV_ERR_INVALID_ARG


def test_decode_rejects_invalid_arguments(lib):
    s = shape()
    dec = lambda **kw: S.selkv_decode_attn(
        kw.get("shape", s), kw.get("q", FAKE), FAKE, FAKE, kw.get("bias", FAKE), FAKE,
        kw.get("k_new", None), kw.get("v_new", None), FAKE, kw.get("ws", FAKE),
        kw.get("wsb", 1 << 40), 0)
    assert dec(q=0) == S.SELKV_ERR_INVALID_ARG
    assert dec(k_new=FAKE) == S.SELKV_ERR_INVALID_ARG          # k_new without v_new
    assert dec(bias=FAKE + 4) == S.SELKV_ERR_INVALID_ARG
    assert dec(shape=shape(head_dim=80)) == S.SELKV_ERR_UNSUPPORTED
    assert dec(shape=shape(m_cap=0)) == S.SELKV_ERR_INVALID_ARG
    assert dec(ws=0) == S.SELKV_ERR_WORKSPACE
    assert dec(wsb=100) == S.SELKV_ERR_WORKSPACE


def test_score_rejects_invalid_arguments(lib):
    s = shape()
    ws_size = S.selkv_score_workspace_size(s)
    assert ws_size > 256 and ws_size % 256 == 0 and ws_size < S.selkv_compress_workspace_size(s)
    assert S.selkv_score_workspace_size(shape(num_kv_heads=7)) == 0
    sc = lambda **kw: S.selkv_score(kw.get("shape", s), kw.get("n_len", [16384]), kw.get("K", FAKE), FAKE,
                                    kw.get("attn", FAKE), kw.get("passes", S.SELKV_SCORE_ALL),
                                    kw.get("ws", FAKE), kw.get("wsb", 1 << 40), 0)
    assert sc(passes=0) == S.SELKV_ERR_INVALID_ARG
    assert sc(passes=4) == S.SELKV_ERR_INVALID_ARG
    assert sc(n_len=[40]) == S.SELKV_ERR_INVALID_ARG           # W = 64 > n_b
    assert sc(n_len=[20000]) == S.SELKV_ERR_INVALID_ARG        # n_b > n_cap
    assert sc(K=0) == S.SELKV_ERR_INVALID_ARG
    assert sc(K=FAKE + 8) == S.SELKV_ERR_INVALID_ARG
    assert sc(attn=0) == S.SELKV_ERR_INVALID_ARG               # the column sums need an output
    assert sc(attn=0, passes=S.SELKV_SCORE_COLSUMS) == S.SELKV_ERR_INVALID_ARG
    assert sc(shape=shape(head_dim=96)) == S.SELKV_ERR_UNSUPPORTED
    assert sc(ws=0) == S.SELKV_ERR_WORKSPACE
    assert sc(wsb=ws_size - 256) == S.SELKV_ERR_WORKSPACE
    # the row-statistics pass alone writes no attention: a NULL output passes validation
    # (checked with a workspace too small, so that nothing is launched)
    assert sc(attn=0, passes=S.SELKV_SCORE_ROWSTATS, wsb=16) == S.SELKV_ERR_WORKSPACE


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    import paper_2607_16213_gb300._binding as bind
    monkeypatch.setattr(bind, "_LIB", None)
    monkeypatch.setattr(bind, "library_path", lambda: str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        bind.library()
