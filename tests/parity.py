"""GPU-vs-oracle comparison helpers for the parity tests.

Discrete decisions (per-KV-head top-k, trim, routing, merge/drop) must agree exactly.  The
margin rule allows one exception: where the oracle's own margin at a decision is below the
arithmetic noise of the fp32 GPU path, either resolution is correct; the check then verifies
that the GPU's choice is one of the near-tied options and the oracle continues from the GPU's
choice ("follow"), so the continuous outputs downstream are still compared element by
element.  Every such follow is counted (`*_near_ties`), and check_sequence fails when a
sequence has more than `max_near_ties` of them (default 0: every decision exact).

Beside the counts, the oracle's smallest margin at each kind of decision boundary is recorded
(`*_min_gap`: the relative gap between the last value taken and the first one left out of a
top-k or trim, between the best and the runner-up kept `a` of a routing bucket; the smallest
|sim| of a routed evicted token), which shows how close to a tie the exact agreements came.
With SELKV_PARITY_LOG set, each checked sequence appends one JSON line (test id, workload,
sequence, counts and margins) to that file.

Margins (derived from the arithmetic of the GPU path):
  DELTA      relative gap on scores / cumulative attention: the rule's ambiguity margin,
             1e-5.  The fp32 GPU values of `a` and of the pooled scores carry a relative error
             of at most ~4e-6 on every workload checked (fp32 sums of exponentials whose
             arguments carry rounding error), so a gap of 1e-5 cannot be reordered by that
             noise: two values each off by 4e-6 relative keep their order.
  DELTA_SIM  absolute margin on the cosine around 0 (merge vs drop).
  DELTA_COS  absolute margin between two cosines (full cosine routing): the GPU's cosines are
             fp32 sums of d products (exact for bf16 inputs), a few 1e-7 off the exact value.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
import torch

import synth
from oracle import selkv_oracle as O
from paper_2607_16213_gb300 import api
import paper_2607_16213_gb300 as S

DELTA = 1e-5
DELTA_SIM = 1e-5
DELTA_COS = 1e-5

# continuous tolerances
ATTN_RTOL = 5e-5        # a and pooled scores: relative to the value (plus a tiny floor)
GATE_ATOL = 2e-6        # g on the same target
RATIO_RTOL = 2e-5       # R
BIAS_ATOL = 2e-5        # alpha * ln(mean R)
VC_FP32_RTOL = 2e-5     # merged values, fp32 storage
DEC_BF16_MAX, DEC_BF16_MEAN = 2e-2, 2e-3   # decode: bf16 storage, fp32 accumulation
DEC_FP32_REL = 1e-5     # decode: fp32 storage, relative to max |out|


def device():
    return torch.device("cuda:0")


def to_dev(x: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x)).to(device())
    return t.to(torch.bfloat16) if dtype == "bf16" else t


def params_of(p: O.Params) -> S.selkv_params:
    return S.selkv_params(alpha=p.alpha, pool_kernel=p.pool_kernel, bucket=p.bucket,
                          recent=p.recent, gate_mode=p.gate_mode, empty_bucket=p.empty_bucket,
                          select_mode=p.select_mode, rope=p.rope, rope_theta=p.rope_theta,
                          bias_mode=p.bias_mode, routing=p.routing)


def run_compress(wl: synth.Workload, x: dict, p: O.Params, rho=None, extra: int = 0):
    rho = wl.rho if rho is None else rho
    n_len = [int(v) for v in x["n_len"]]
    m_cap = api.capacity(max(n_len), rho, extra=extra)
    shape = api.make_shape(wl.dtype, wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                           wl.obs_window, wl.n, m_cap)
    K, V, Q = to_dev(x["K"], wl.dtype), to_dev(x["V"], wl.dtype), to_dev(x["Q_obs"], wl.dtype)
    ws = api.Workspace(S.selkv_compress_workspace_size(shape))
    cache = api.compress(shape, n_len, rho, K, V, Q, params=params_of(p), debug=True, workspace=ws)
    torch.cuda.synchronize()
    flags = ws.errors()
    assert flags == 0, "device error flags %#x" % flags
    host = {k: v.cpu().numpy() for k, v in cache.debug.items()}
    host["K_c"] = cache.K_c.float().cpu().numpy()
    host["V_c"] = cache.V_c.float().cpu().numpy()
    host["bias"] = cache.bias.cpu().numpy()
    host["lengths"] = cache.lengths.cpu().numpy()
    return cache, host, (K, V, Q)


def boundary_gap(values: np.ndarray, k: int) -> float:
    """The oracle's margin at a top-k boundary: relative gap between the k-th largest value
    and the next one (inf when nothing is left out)."""
    if k <= 0 or k >= values.size:
        return math.inf
    part = -np.partition(-values, (k - 1, k))
    hi, lo = float(part[k - 1]), float(part[k])
    return (hi - lo) / max(abs(hi), 1e-300)


def check_topk_choice(gpu_mask: np.ndarray, values: np.ndarray, k: int, what: str) -> int:
    """GPU top-k equals the oracle's up to swaps among near-ties of the k-th value."""
    assert int(gpu_mask.sum()) == k, "%s: %d selected, expected %d" % (what, gpu_mask.sum(), k)
    own = O.top_k_mask(values, k)
    diff = np.flatnonzero(gpu_mask != own)
    if diff.size == 0:
        return 0
    thr = np.sort(values)[::-1][k - 1]
    gap = np.abs(values[diff] - thr) / max(abs(thr), 1e-300)
    assert gap.max() <= DELTA, "%s: %d positions differ, largest gap %.3g" % (what, diff.size, gap.max())
    return int(diff.size)


NEAR_TIE_KEYS = ("topk_near_ties", "trim_near_ties", "route_near_ties", "decision_near_ties")


class Stats(dict):
    def add(self, k, v=1):
        self[k] = self.get(k, 0) + v

    def low(self, k, v):
        """Keep the smallest value seen under k."""
        self[k] = min(self.get(k, math.inf), float(v))

    def near_ties(self) -> int:
        return sum(int(self.get(k, 0)) for k in NEAR_TIE_KEYS)


def _log(wl, b: int, st: Stats):
    path = os.environ.get("SELKV_PARITY_LOG")
    if not path:
        return
    test = os.environ.get("PYTEST_CURRENT_TEST", "").rsplit(" ", 1)[0]
    rec = {"test": test, "workload": wl.name, "seq": b}
    rec.update({k: (None if isinstance(v, float) and math.isinf(v) else v) for k, v in st.items()})
    with open(path, "a") as f:
        f.write(json.dumps(rec) + "\n")


def route_gap(a_kv: np.ndarray, kept: np.ndarray, bucket: int) -> float:
    """The oracle's smallest routing margin in one KV head: over the buckets that evict at
    least one token and keep two or more, the relative gap between the largest kept `a` and
    the runner-up (inf when there is no such bucket)."""
    n = kept.size
    nb = (n + bucket - 1) // bucket
    kp = np.flatnonzero(kept)
    ev_b = np.zeros(nb, dtype=bool)
    ev_b[np.flatnonzero(~kept) // bucket] = True
    bk = kp // bucket
    sel = ev_b[bk]
    kp, bk = kp[sel], bk[sel]
    if kp.size < 2:
        return math.inf
    order = np.lexsort((-a_kv[kp], bk))
    kp, bk = kp[order], bk[order]
    first = np.ones(kp.size, dtype=bool)
    first[1:] = bk[1:] != bk[:-1]
    second = np.zeros(kp.size, dtype=bool)
    second[1:] = first[:-1] & ~first[1:]
    if not second.any():
        return math.inf
    top = a_kv[kp[np.flatnonzero(second) - 1]]
    run = a_kv[kp[second]]
    return float(((top - run) / np.maximum(np.abs(top), 1e-300)).min())


def check_sequence(wl, x, host, b: int, p: O.Params, rho=None, stats: Stats = None,
                   max_near_ties: int = 0) -> dict:
    """Compare sequence b of one compressed layer with the oracle, stage by stage.  Fails when
    the sequence needed more than `max_near_ties` follows of the margin rule; the sequence's
    counts and margins are added to `stats` and logged (SELKV_PARITY_LOG)."""
    seq = Stats()
    out = _check_sequence(wl, x, host, b, p, wl.rho if rho is None else rho, seq)
    _log(wl, b, seq)
    if stats is not None:
        for k, v in seq.items():
            if k.endswith("_max"):
                stats[k] = max(stats.get(k, 0.0), v)
            elif k.endswith("_min_gap"):
                stats.low(k, v)
            else:
                stats.add(k, v)
    assert seq.near_ties() <= max_near_ties, \
        "sequence %d: %d decisions resolved by the margin rule (%s)" % (
            b, seq.near_ties(), {k: seq.get(k, 0) for k in NEAR_TIE_KEYS})
    return out


def _check_sequence(wl, x, host, b: int, p: O.Params, rho: float, stats: Stats) -> dict:
    n = int(x["n_len"][b])
    K = x["K"][b, :, :n].astype(np.float64)
    V = x["V"][b, :, :n].astype(np.float64)
    Q = x["Q_obs"][b].astype(np.float64)
    Hkv = K.shape[0]
    m, m_s = O.budget(n, rho, p.recent)
    assert int(host["lengths"][b]) == m
    n_cand = n - p.recent

    # Sec. 3.1 / Eq. 1: cumulative attention and pooled contribution score (continuous)
    a = O.cumulative_attention(Q, K, n)
    vn = O.value_norms(V, n)
    cp = O.pool_scores(a * vn, n_cand, p.pool_kernel)
    a_g = host["attn"][b, :, :n].astype(np.float64)
    err_a = np.abs(a_g - a) / (np.abs(a) + 1e-30)
    stats["attn_rel_max"] = max(stats.get("attn_rel_max", 0.0), float(err_a.max()))
    assert err_a.max() <= ATTN_RTOL, "attention rel err %.3g" % err_a.max()
    sc_g = host["score"][b, :, :n_cand].astype(np.float64)
    err_s = np.abs(sc_g - cp) / (np.abs(cp) + 1e-30)
    stats["score_rel_max"] = max(stats.get("score_rel_max", 0.0), float(err_s.max()))
    assert err_s.max() <= ATTN_RTOL, "score rel err %.3g" % err_s.max()

    # Eq. 2: each KV head's top-m_s
    per_kv = host["topk"][b, :, :n_cand].astype(bool)
    if m_s > 0:
        for kv in range(Hkv):
            stats.add("topk_near_ties", check_topk_choice(per_kv[kv], cp[kv], m_s, "top-k kv%d" % kv))
            stats.low("topk_min_gap", boundary_gap(cp[kv], m_s))
    else:
        assert not per_kv.any()
    if p.select_mode == O.SELECT_PER_HEAD:
        return _check_per_head(wl, x, host, b, p, stats, n, m, m_s, K, V, a, per_kv)
    # Sec. 3.3: union and trim, continuing from the GPU's per-head choice
    sel = O.select_shared(cp, n, m_s, p.recent, follow_per_kv=per_kv)
    kept_idx_g = host["kept_idx"][b, :m].astype(np.int64)
    assert (np.diff(kept_idx_g) > 0).all() and kept_idx_g.min() >= 0 and kept_idx_g.max() < n
    kept_g = np.zeros(n, dtype=bool)
    kept_g[kept_idx_g] = True
    assert kept_g[n - p.recent:].all()
    if sel.trimmed:
        members = np.flatnonzero(sel.union)
        mean = cp.mean(axis=0)
        gpu_in = kept_g[:n_cand][members]
        stats.add("trim_near_ties", check_topk_choice(gpu_in, mean[members], m_s, "trim"))
        stats.low("trim_min_gap", boundary_gap(mean[members], m_s))
        assert not kept_g[:n_cand][~sel.union].any(), "kept a candidate outside the union"
    else:
        assert (kept_g[:n_cand] == sel.union).all()

    # Eq. 3-6 per KV head, continuing from the GPU's kept set
    tgt_g = host["target"][b, :, :n].astype(np.int64)
    gate_g = host["gate"][b, :, :n].astype(np.float64)
    dec_g = host["decision"][b, :, :n]
    Vc_o = np.empty((Hkv, m, V.shape[2]))
    R_o = np.empty((Hkv, m))
    for kv in range(Hkv):
        g_o = _check_route_gate(p, stats, kv, n, a[kv], V[kv], kept_g, tgt_g[kv], gate_g[kv], dec_g[kv])
        Vc_o[kv], R_o[kv] = O.merge(a[kv], V[kv], kept_idx_g, tgt_g[kv], g_o)
    if p.bias_mode == O.BIAS_COUNT:   # counts from the GPU's own targets and gates
        M = np.stack([O.merge_counts(kept_idx_g, tgt_g[kv], gate_g[kv]) for kv in range(Hkv)])
        bias_o = O.count_bias(M, p.alpha, per_head=False)
    else:
        bias_o = O.gqa_bias(R_o, p.alpha)

    # continuous outputs
    for kv in range(Hkv):
        check_keys(host["K_c"][b, kv, :m], K[kv, kept_idx_g], kept_idx_g, p, wl.dtype)
    R_g = host["ratio"][b, :, :m].astype(np.float64)
    err_r = np.abs(R_g - R_o) / R_o
    stats["ratio_rel_max"] = max(stats.get("ratio_rel_max", 0.0), float(err_r.max()))
    assert err_r.max() <= RATIO_RTOL, "R rel err %.3g" % err_r.max()
    bias_g = host["bias"][b, :, :m].astype(np.float64)
    assert (bias_g == bias_g[:1]).all(), "bias rows differ across KV heads"
    err_b = np.abs(bias_g[0] - bias_o)
    stats["bias_abs_max"] = max(stats.get("bias_abs_max", 0.0), float(err_b.max()))
    assert err_b.max() <= BIAS_ATOL, "bias err %.3g" % err_b.max()
    Vc_g = host["V_c"][b, :, :m].astype(np.float64)
    if wl.dtype == "bf16":
        # the GPU rounds its fp32 result to bf16 once: within one bf16 rounding of the exact
        # value (half an ulp, 2^-9 relative), plus fp32 noise
        tol = np.abs(Vc_o) * 2.0 ** -8 + 1e-5
    else:
        tol = np.abs(Vc_o) * VC_FP32_RTOL + 1e-6
    err_v = np.abs(Vc_g - Vc_o) - tol
    assert err_v.max() <= 0, "V_c error beyond tolerance by %.3g" % err_v.max()
    return dict(n=n, m=m, K_c=K[:, kept_idx_g], V_c=Vc_o, bias=bias_o, a=a, kept_idx=kept_idx_g)


def check_keys(host_Kc: np.ndarray, K_kept: np.ndarray, kept_idx: np.ndarray, p: O.Params, dtype: str):
    """K_c rows of one KV head: the kept keys unchanged, or with RoPE repositioning (Eq. 7) the
    oracle's re-embedded keys within one rounding to the storage type plus fp32 angle error
    (4e-6 of the row norm)."""
    if p.rope == O.ROPE_OFF:
        np.testing.assert_array_equal(host_Kc, K_kept.astype(np.float32))
        return
    want = O.reposition(K_kept, kept_idx, p.rope_theta, p.rope)
    rel = 2.0 ** -8 if dtype == "bf16" else 0.0
    tol = np.abs(want) * rel + 4e-6 * np.linalg.norm(want, axis=1, keepdims=True)
    err = np.abs(host_Kc.astype(np.float64) - want) - tol
    assert err.max() <= 0, "repositioned keys beyond tolerance by %.3g" % err.max()


def _cos(x: np.ndarray, y: np.ndarray) -> float:
    den = math.sqrt(float(x @ x)) * math.sqrt(float(y @ y))
    return float(x @ y) / den if den > 0 else 0.0


def _check_routing(p, stats, a_kv, V_kv, kept_g, tgt_g, ev):
    """Routing (Eq. 3) of one KV head: the GPU's targets against the oracle's, exact except at near
    ties (bucket routing: the same ring distance and a within DELTA; cosine routing: cosines
    within DELTA_COS)."""
    if p.routing == O.ROUTE_COSINE:
        own = O.route_cosine(V_kv, kept_g)
    else:
        own = O.route(a_kv, kept_g, p.bucket, p.empty_bucket)
    diff = ev[tgt_g[ev] != own[ev]]
    for j in diff:
        tg, to = int(tgt_g[j]), int(own[j])
        assert tg >= 0 and to >= 0 and kept_g[tg], "target of %d: gpu %d oracle %d" % (j, tg, to)
        if p.routing == O.ROUTE_COSINE:
            assert _cos(V_kv[j], V_kv[to]) - _cos(V_kv[j], V_kv[tg]) <= DELTA_COS, "routing differs at %d" % j
        else:
            # same ring distance, a within DELTA of the oracle's choice
            assert abs(tg // p.bucket - j // p.bucket) == abs(to // p.bucket - j // p.bucket)
            assert abs(a_kv[tg] - a_kv[to]) <= DELTA * a_kv[to], "routing differs at %d" % j
    stats.add("route_near_ties", int(diff.size))
    if p.routing != O.ROUTE_COSINE:
        stats.low("route_min_gap", route_gap(a_kv, kept_g, p.bucket))


def _check_route_gate(p, stats, kv, n, a_kv, V_kv, kept_g, tgt_g, gate_g, dec_g):
    """Routing, gate and decision of one KV head against the oracle, continuing from the
    GPU's kept set; returns the oracle's gates for that head's merge."""
    ev = np.flatnonzero(~kept_g)
    assert (tgt_g[kept_g] == -1).all() and (dec_g[kept_g] == 2).all()
    _check_routing(p, stats, a_kv, V_kv, kept_g, tgt_g, ev)
    g_o, sim_o, dec_o = O.gate(V_kv, tgt_g, p.gate_mode)
    routed = ev[tgt_g[ev] >= 0]
    err_g = np.abs(gate_g[routed] - g_o[routed])
    stats["gate_abs_max"] = max(stats.get("gate_abs_max", 0.0), float(err_g.max(initial=0.0)))
    assert err_g.max(initial=0.0) <= GATE_ATOL, "gate err %.3g" % err_g.max()
    ddiff = ev[dec_g[ev] != dec_o[ev]]
    assert (np.abs(sim_o[ddiff]) <= DELTA_SIM).all(), "merge/drop differs away from sim = 0"
    stats.add("decision_near_ties", int(ddiff.size))
    if routed.size and p.gate_mode == O.GATE_COSINE:
        stats.low("sim_min_abs", np.abs(sim_o[routed]).min())
    stats.add("evicted", int(ev.size))
    stats.add("merged", int((dec_g[ev] == 1).sum()))
    return g_o


def _check_values(wl, host, b, m, Vc_o, what="V_c"):
    Vc_g = host["V_c"][b, :, :m].astype(np.float64)
    if wl.dtype == "bf16":
        tol = np.abs(Vc_o) * 2.0 ** -8 + 1e-5
    else:
        tol = np.abs(Vc_o) * VC_FP32_RTOL + 1e-6
    err_v = np.abs(Vc_g - Vc_o) - tol
    assert err_v.max() <= 0, "%s error beyond tolerance by %.3g" % (what, err_v.max())


def _check_per_head(wl, x, host, b, p, stats, n, m, m_s, K, V, a, per_kv):
    """Per-head mode (Sec. 3.3 per-head selection, Sec. 3.6 per-head bias): each KV head's
    kept set is its own top-m_s plus the recent window; Eq. 3-6 and the bias per head."""
    Hkv, n_cand = K.shape[0], n - p.recent
    tgt_g = host["target"][b, :, :n].astype(np.int64)
    gate_g = host["gate"][b, :, :n].astype(np.float64)
    dec_g = host["decision"][b, :, :n]
    Vc_o = np.empty((Hkv, m, V.shape[2]))
    R_o = np.empty((Hkv, m))
    kept_idx_g = host["kept_idx"][b, :, :m].astype(np.int64)
    for kv in range(Hkv):
        kept_g = np.zeros(n, dtype=bool)
        kept_g[kept_idx_g[kv]] = True
        assert (np.diff(kept_idx_g[kv]) > 0).all() and int(kept_g.sum()) == m
        expect = per_kv[kv].copy() if m_s > 0 else np.zeros(n_cand, dtype=bool)
        assert (kept_g[:n_cand] == expect).all() and kept_g[n_cand:].all(), "head %d kept set" % kv
        g_o = _check_route_gate(p, stats, kv, n, a[kv], V[kv], kept_g, tgt_g[kv], gate_g[kv], dec_g[kv])
        Vc_o[kv], R_o[kv] = O.merge(a[kv], V[kv], kept_idx_g[kv], tgt_g[kv], g_o)
        check_keys(host["K_c"][b, kv, :m], K[kv, kept_idx_g[kv]], kept_idx_g[kv], p, wl.dtype)
    if p.bias_mode == O.BIAS_COUNT:
        M = np.stack([O.merge_counts(kept_idx_g[kv], tgt_g[kv], gate_g[kv]) for kv in range(Hkv)])
        bias_o = O.count_bias(M, p.alpha, per_head=True)
    else:
        bias_o = O.per_head_bias(R_o, p.alpha)
    R_g = host["ratio"][b, :, :m].astype(np.float64)
    err_r = np.abs(R_g - R_o) / R_o
    stats["ratio_rel_max"] = max(stats.get("ratio_rel_max", 0.0), float(err_r.max()))
    assert err_r.max() <= RATIO_RTOL, "R rel err %.3g" % err_r.max()
    err_b = np.abs(host["bias"][b, :, :m].astype(np.float64) - bias_o)
    stats["bias_abs_max"] = max(stats.get("bias_abs_max", 0.0), float(err_b.max()))
    assert err_b.max() <= BIAS_ATOL, "bias err %.3g" % err_b.max()
    _check_values(wl, host, b, m, Vc_o)
    K_c = np.stack([K[kv, kept_idx_g[kv]] for kv in range(Hkv)])
    return dict(n=n, m=m, K_c=K_c, V_c=Vc_o, bias=bias_o, a=a, kept_idx=kept_idx_g)


def check_decode(out_gpu: np.ndarray, want: np.ndarray, dtype: str, what: str = "decode"):
    err = np.abs(out_gpu.astype(np.float64) - want)
    if dtype == "bf16":
        assert err.max() <= DEC_BF16_MAX, "%s max-abs %.3g" % (what, err.max())
        assert err.mean() <= DEC_BF16_MEAN, "%s mean-abs %.3g" % (what, err.mean())
    else:
        rel = err.max() / max(np.abs(want).max(), 1e-30)
        assert rel <= DEC_FP32_REL, "%s rel %.3g" % (what, rel)
    return float(err.max()), float(err.mean())


def check_properties(wl, x, host, p: O.Params, rho=None):
    """Structural checks of every sequence of a compressed layer that hold at any size:
    exactly m_b kept positions in ascending order including the recent window, every evicted
    token routed to a kept token of its own bucket when that bucket keeps one (Eq. 3), merge
    decisions consistent with g (Eq. 4), R >= 1 and R = 1 for kept tokens that are nobody's
    target, bias = alpha ln(mean over KV heads of R) (Sec. 3.6), keys copied unchanged, and
    the values of kept tokens that absorbed nothing copied unchanged."""
    rho = wl.rho if rho is None else rho
    for b in range(wl.batch):
        n = int(x["n_len"][b])
        m, m_s = O.budget(n, rho, p.recent)
        assert int(host["lengths"][b]) == m
        kept_idx = host["kept_idx"][b, :m].astype(np.int64)
        assert (np.diff(kept_idx) > 0).all() and kept_idx[0] >= 0 and kept_idx[-1] < n
        kept = np.zeros(n, dtype=bool)
        kept[kept_idx] = True
        assert kept[n - p.recent:].all()
        bucket_has = np.add.reduceat(kept.astype(np.int64), np.arange(0, n, p.bucket)) > 0
        ev = np.flatnonzero(~kept)
        tgt = host["target"][b, :, :n].astype(np.int64)
        dec = host["decision"][b, :, :n]
        g = host["gate"][b, :, :n]
        R = host["ratio"][b, :, :m].astype(np.float64)
        for kv in range(wl.num_kv_heads):
            t = tgt[kv, ev]
            assert (t >= 0).all() and kept[t].all(), "evicted token without a kept target"
            own = bucket_has[ev // p.bucket]
            assert (t[own] // p.bucket == ev[own] // p.bucket).all(), "target outside the bucket"
            assert ((g[kv, ev] > 0) == (dec[kv, ev] == 1)).all() and (dec[kv, kept] == 2).all()
            assert (g[kv, ev] >= 0).all() and (g[kv, ev] <= 1).all()
            assert (R[kv] >= 1.0).all()
            absorbed = np.zeros(n, dtype=bool)
            absorbed[t[g[kv, ev] > 0]] = True
            slot_abs = absorbed[kept_idx]
            assert (R[kv][~slot_abs] == 1.0).all()
            np.testing.assert_array_equal(host["K_c"][b, kv, :m], x["K"][b, kv, kept_idx])
            np.testing.assert_array_equal(host["V_c"][b, kv, :m][~slot_abs], x["V"][b, kv, kept_idx][~slot_abs])
        want_bias = p.alpha * np.log(R.mean(axis=0))
        bias = host["bias"][b, :, :m].astype(np.float64)
        assert (bias == bias[:1]).all()
        np.testing.assert_allclose(bias[0], want_bias, rtol=1e-6, atol=1e-6)
