"""SelKV oracle: a plain, slow, fp64 CPU statement of what SelKV computes.

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
leg may import or call this module.  The CUDA library never calls it and shares no code with
it; the two meet only at the seeded inputs of the `synth` module.

What it follows (arxiv 2607.16213, "SelKV: Selective KV Cache Merging with Per-Token
Merge-or-Drop and Attention Compensation"):

  observation re-pass (Sec. 3.1) -> contribution score (Eq. 1) -> average pooling (Sec. 3.2)
  -> budget m = floor(rho n), recent window m_r (Sec. 3.1) -> per-KV-head top-m_s, union over
  KV heads, trim by mean score (Eq. 2, Sec. 3.3 "Union selection"; or, in per-head mode,
  each head's own top-m_s, Sec. 3.3 "Per-head selection") -> bucket-attention routing
  (Eq. 3, Sec. 3.4) -> soft cosine gate (Eq. 4, Sec. 3.5) -> gated attention-weighted merge (Eq. 5) -> attention
  ratio (Eq. 6) -> GQA bias alpha*log(mean_kv R) (Sec. 3.6) -> decode with the bias (Alg. 1,
  last step).  RoPE repositioning (Eq. 7, Sec. 3.7) is off by default, as in the paper's
  configuration (Sec. 4.1), and available as a parameter (R18).

Readings where the paper is silent or garbled (each is a named choice, mirrored by the CUDA
path):
  R1  the re-pass is causal: window row i sits at position p_i = n - W + i and sees j <= p_i.
  R2  softmax scale 1/sqrt(d).
  R3  query head h uses KV head h // G.
  R4  per-KV-head scores and cumulative attention are the mean over the G query heads;
      then c_kv = a_kv * ||v_kv|| (Eq. 1 averaged over the group).
  R5  pooling: stride 1, zero padding, divide by the kernel size, over the candidate range
      [0, n - m_r) only (recent-window scores are not pooled in).
  R6  m = floor(rho * n) in double; m_s = m - m_r must be >= 0.
  R7  every top-k, trim and argmax orders by value descending, then index ascending.
  R8  trim key = mean over KV heads of the pooled per-KV-head score, restricted to the union.
  R9  Eq. 3's argmax uses a_{kv,i}, the cumulative observation-window attention paid to the
      candidate i (the paper says the lookup uses the window queries' attention); so every
      evicted token of a bucket shares one target per KV head.
  R10 bucket(j) = floor(j / B) from position 0; the last bucket may be partial.
  R11 empty bucket: "expand" looks at the kept tokens of buckets b-r and b+r for r = 1, 2, ...
      and takes the first non-empty ring; "drop" gives those tokens g = 0 and no target.
  R12 only values are merged; kept keys are unchanged.
  R13 the gate uses the original (pre-merge) target value; a zero norm gives sim = 0; g is
      clamped to [0, 1].
  R14 decision MERGE iff g > 0, else DROP.
  R15 a_i = 0 guard: R = 1, and v~ = v_i when the denominator is 0.
  R16 GQA bias = alpha * ln(mean over KV heads of R) (natural log), per layer.
  R17 per-head mode (Sec. 3.3, MHA models; Sec. 3.6 "per head without cross-head
      averaging"): each KV head keeps its own top-m_s of its pooled score plus the recent
      window, routes, gates and merges against that set, and its bias is alpha * ln R of its
      own entries.  On a GQA model the G query heads of a KV head share its set.
  R18 RoPE repositioning (Eq. 7, off by default as in Sec. 4.1): the kept key of slot s,
      originally at position p_old = its index in the sequence, is re-embedded at p_new = s.
      RoPE is the plain rotary embedding with base theta: frequency f in [0, d/2) rotates the
      pair (k[f], k[f + d/2]) ("half" layout) or (k[2f], k[2f + 1]) ("interleaved" layout) by
      the angle p * theta^(-2f/d).  Values are not rotated.
  R19 count bias (the KeepKV compensation Sec. 3.6 replaces, kept as a variant): M_i = number
      of evicted tokens merged into kept token i (routed to i with g > 0); bias = alpha *
      ln(1 + mean over KV heads of M_i) in the shared mode, alpha * ln(1 + M_{h,i}) per head
      in the per-head mode (alpha = 1 is KeepKV's log(1 + M_i)).
  R20 full cosine routing (the alternative Sec. 3.4 prices at O(H |S| |E| d)): pi(j) is the
      kept token of the head with the largest cos(v_j, v_i) over all kept tokens, with the
      original (pre-merge) values; ties to the lower position; a zero norm gives cosine 0.
  R21 compensation averaged across layers (the overview of Sec. 3 offers it next to the per-
      layer bias): one value per (sequence, position), shared by every layer, is the mean over
      the L layers of the layer's per-slot quantity at that position (the KV-head mean R of
      R16, or M of R19; per KV head in the per-head mode), a layer that evicted the position
      counting the neutral value (R = 1, M = 0); every layer's slot holding the position then
      gets alpha * ln(mean R), or alpha * ln(1 + mean M).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional

import numpy as np

GATE_COSINE, GATE_OPEN, GATE_CLOSED = 0, 1, 2
SELECT_SHARED, SELECT_PER_HEAD = 0, 1
ROPE_OFF, ROPE_HALF, ROPE_INTERLEAVED = 0, 1, 2
BIAS_RATIO, BIAS_COUNT = 0, 1
ROUTE_BUCKET, ROUTE_COSINE = 0, 1
EMPTY_EXPAND, EMPTY_DROP = 0, 1
DECISION_DROP, DECISION_MERGE = 0, 1


@dataclass
class Params:
    """Method hyperparameters (Sec. 4.1 / App. F defaults)."""
    alpha: float = 0.5
    pool_kernel: int = 5
    bucket: int = 32
    recent: int = 16
    gate_mode: int = GATE_COSINE
    empty_bucket: int = EMPTY_EXPAND
    select_mode: int = SELECT_SHARED
    rope: int = ROPE_OFF
    rope_theta: float = 10000.0
    bias_mode: int = BIAS_RATIO
    routing: int = ROUTE_BUCKET


# ----------------------------------------------------------------------------------------
# Sec. 3.1: budget
# ----------------------------------------------------------------------------------------
def budget(n: int, rho: float, recent: int):
    """m = floor(rho * n) kept entries; the last m_r = recent are always kept; m_s = m - m_r
    are chosen by score (Sec. 3.1, reading R6)."""
    m = int(math.floor(float(rho) * float(n)))
    return m, m - recent


# ----------------------------------------------------------------------------------------
# Sec. 3.1 two-pass re-pass + Eq. 1: observation-window attention
# ----------------------------------------------------------------------------------------
def observation_attention(Q: np.ndarray, K: np.ndarray, n: int) -> np.ndarray:
    """A[h, i, j]: softmax over keys j <= p_i of q_{h,i} . k_{kv(h),j} / sqrt(d), for the W
    window rows i at positions p_i = n - W + i (Sec. 3.1; readings R1-R3).

    Q: [Hq][W][d], K: [Hkv][>=n][d] (float64).  Returns [Hq][W][n]."""
    Hq, W, d = Q.shape
    Hkv = K.shape[0]
    G = Hq // Hkv
    A = np.zeros((Hq, W, n))
    pos = n - W + np.arange(W)
    visible = np.arange(n)[None, :] <= pos[:, None]
    for h in range(Hq):
        s = (Q[h] @ K[h // G, :n].T) / math.sqrt(d)
        s = np.where(visible, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        e = np.exp(s)
        A[h] = e / e.sum(axis=1, keepdims=True)
    return A


def cumulative_attention(Q: np.ndarray, K: np.ndarray, n: int) -> np.ndarray:
    """a[kv, j] = (1/G) sum_{h in group(kv)} sum_i A[h, i, j] (Eq. 5's a, averaged over the
    query group, reading R4).  Computed one query head at a time.  Returns [Hkv][n]."""
    Hq, W, d = Q.shape
    Hkv = K.shape[0]
    G = Hq // Hkv
    a = np.zeros((Hkv, n))
    for h in range(Hq):
        A_h = observation_attention(Q[h:h + 1], K[h // G:h // G + 1], n)[0]
        a[h // G] += A_h.sum(axis=0)
    return a / G


def value_norms(V: np.ndarray, n: int) -> np.ndarray:
    """||v_{kv,j}||_2 for j < n.  V: [Hkv][>=n][d]."""
    return np.sqrt((V[:, :n] ** 2).sum(axis=2))


def contribution_scores(a: np.ndarray, V: np.ndarray, n: int) -> np.ndarray:
    """Eq. 1 per KV head: c[kv, j] = a[kv, j] * ||v_{kv,j}|| (reading R4)."""
    return a * value_norms(V, n)


def pool_scores(c: np.ndarray, n_cand: int, kernel: int) -> np.ndarray:
    """Average pooling of the scores over the candidate range [0, n_cand) (Sec. 3.2,
    reading R5): out[j] = (1/kernel) * sum_{|t| <= kernel//2} c[j + t], with terms outside
    [0, n_cand) taken as zero.  c: [Hkv][>=n_cand].  Returns [Hkv][n_cand]."""
    half = kernel // 2
    out = np.zeros((c.shape[0], n_cand))
    idx = np.arange(n_cand)
    for t in range(-half, half + 1):
        src = idx + t
        ok = (src >= 0) & (src < n_cand)
        out[:, ok] += c[:, src[ok]]
    return out / kernel


# ----------------------------------------------------------------------------------------
# Eq. 2 + Sec. 3.3: selection
# ----------------------------------------------------------------------------------------
def top_k_mask(values: np.ndarray, k: int) -> np.ndarray:
    """Boolean mask of the k best entries: larger value first, then lower index (R7)."""
    order = np.lexsort((np.arange(values.shape[0]), -values))
    mask = np.zeros(values.shape[0], dtype=bool)
    mask[order[:k]] = True
    return mask


@dataclass
class Selection:
    per_kv: np.ndarray        # [Hkv][n_cand] bool: each KV head's top-m_s (Eq. 2)
    union: np.ndarray         # [n_cand] bool
    kept_cand: np.ndarray     # [n_cand] bool: union, trimmed to m_s by mean score (Sec. 3.3)
    kept: np.ndarray          # [n] bool: kept_cand plus the recent window
    trimmed: bool


def select_shared(c_pooled: np.ndarray, n: int, m_s: int, recent: int,
                  follow_per_kv: Optional[np.ndarray] = None,
                  follow_kept: Optional[np.ndarray] = None) -> Selection:
    """GQA union selection (Eq. 2 per KV head, then Sec. 3.3 union and trim; R7, R8).

    follow_per_kv / follow_kept replace the oracle's own per-KV-head choice / final kept
    set with given ones (used only after a test has checked that they differ from the
    oracle's own choice at near-ties only)."""
    Hkv, n_cand = c_pooled.shape
    if follow_per_kv is not None:
        per_kv = np.asarray(follow_per_kv[:, :n_cand], dtype=bool)
    else:
        per_kv = np.stack([top_k_mask(c_pooled[kv], m_s) for kv in range(Hkv)])
    union = per_kv.any(axis=0)
    trimmed = bool(union.sum() > m_s)
    if trimmed:
        mean = c_pooled.mean(axis=0)
        members = np.flatnonzero(union)
        keep = top_k_mask(mean[members], m_s)
        kept_cand = np.zeros(n_cand, dtype=bool)
        kept_cand[members[keep]] = True
    else:
        kept_cand = union.copy()
    kept = np.zeros(n, dtype=bool)
    kept[:n_cand] = kept_cand
    kept[n - recent:] = True
    if follow_kept is not None:
        kept = np.asarray(follow_kept[:n], dtype=bool).copy()
        kept_cand = kept[:n_cand].copy()
    return Selection(per_kv, union, kept_cand, kept, trimmed)


def select_per_head(c_pooled: np.ndarray, n: int, m_s: int, recent: int,
                    follow_per_kv: Optional[np.ndarray] = None) -> np.ndarray:
    """Per-head selection (Eq. 2; Sec. 3.3 "Per-head selection"; R7, R17): each KV head's
    top-m_s of its pooled score over the candidates, plus the recent window.  Returns the
    kept masks [Hkv][n].  follow_per_kv replaces the top-m_s choices as in select_shared."""
    Hkv, n_cand = c_pooled.shape
    kept = np.zeros((Hkv, n), dtype=bool)
    for kv in range(Hkv):
        if follow_per_kv is not None:
            kept[kv, :n_cand] = np.asarray(follow_per_kv[kv, :n_cand], dtype=bool)
        else:
            kept[kv, :n_cand] = top_k_mask(c_pooled[kv], m_s)
        kept[kv, n - recent:] = True
    return kept


# ----------------------------------------------------------------------------------------
# Eq. 3: bucket-attention routing
# ----------------------------------------------------------------------------------------
def _best(a_kv: np.ndarray, cands: np.ndarray) -> int:
    """argmax of a over candidate positions, ties to the lower position (R7)."""
    best = int(cands[0])
    for i in cands[1:]:
        if a_kv[i] > a_kv[best]:
            best = int(i)
    return best


def route(a_kv: np.ndarray, kept: np.ndarray, bucket: int, empty_policy: int) -> np.ndarray:
    """Merge target pi(j) for every evicted j of one KV head; -1 for kept tokens and for
    tokens left without a target (Eq. 3; readings R9-R11).

    The argmax over the kept tokens of bucket(j) of a_kv does not depend on j, so it is
    found once per bucket."""
    n = kept.shape[0]
    nb = (n + bucket - 1) // bucket
    kept_in = [np.flatnonzero(kept[b * bucket:min(n, (b + 1) * bucket)]) + b * bucket
               for b in range(nb)]
    target = np.full(n, -1, dtype=np.int64)
    for b in range(nb):
        evicted = [j for j in range(b * bucket, min(n, (b + 1) * bucket)) if not kept[j]]
        if not evicted:
            continue
        t = -1
        if kept_in[b].size:
            t = _best(a_kv, kept_in[b])
        elif empty_policy == EMPTY_EXPAND:
            r = 1
            while t < 0 and (b - r >= 0 or b + r < nb):
                ring = []
                if b - r >= 0:
                    ring.extend(kept_in[b - r].tolist())
                if b + r < nb:
                    ring.extend(kept_in[b + r].tolist())
                if ring:
                    t = _best(a_kv, np.array(sorted(ring)))
                r += 1
        for j in evicted:
            target[j] = t
    return target


def route_cosine(V_kv: np.ndarray, kept: np.ndarray) -> np.ndarray:
    """Full cosine routing (R20): every evicted j goes to the kept i with the largest
    cos(v_j, v_i) (ties to the lower i; a zero norm gives cosine 0).  -1 for kept tokens."""
    V_kv = np.asarray(V_kv, dtype=np.float64)
    n = kept.shape[0]
    ki = np.flatnonzero(kept)
    target = np.full(n, -1, dtype=np.int64)
    if ki.size == 0:
        return target
    norms = np.linalg.norm(V_kv[:n], axis=1)
    Vk = V_kv[ki]
    nk = norms[ki]
    for j in np.flatnonzero(~kept):
        cos = np.where((nk > 0) & (norms[j] > 0), (Vk @ V_kv[j]) / np.where(nk > 0, nk, 1.0) /
                       (norms[j] if norms[j] > 0 else 1.0), 0.0)
        target[j] = int(ki[int(np.argmax(cos))])   # argmax keeps the first (lowest) maximum
    return target


# ----------------------------------------------------------------------------------------
# Eq. 4: soft cosine gate
# ----------------------------------------------------------------------------------------
def gate(V_kv: np.ndarray, target: np.ndarray, mode: int):
    """g_j and sim_j for every routed token (Eq. 4; readings R13, R14).  Tokens without a
    target get g = 0.  Returns (g, sim, decision) over positions [0, n)."""
    n = target.shape[0]
    g = np.zeros(n)
    sim = np.zeros(n)
    for j in np.flatnonzero(target >= 0):
        t = int(target[j])
        nj = math.sqrt(float(V_kv[j] @ V_kv[j]))
        nt = math.sqrt(float(V_kv[t] @ V_kv[t]))
        sim[j] = 0.0 if nj == 0.0 or nt == 0.0 else float(V_kv[j] @ V_kv[t]) / (nj * nt)
        if mode == GATE_OPEN:
            g[j] = 1.0
        elif mode == GATE_CLOSED:
            g[j] = 0.0
        else:
            g[j] = min(max(sim[j], 0.0), 1.0)
    decision = (g > 0).astype(np.uint8)
    return g, sim, decision


# ----------------------------------------------------------------------------------------
# Eq. 5 + Eq. 6: gated merge and attention ratio
# ----------------------------------------------------------------------------------------
def merge(a_kv: np.ndarray, V_kv: np.ndarray, kept_idx: np.ndarray, target: np.ndarray,
          g: np.ndarray):
    """For each kept i (in kept_idx order):
         den_i = a_i + sum_{pi(j)=i} g_j a_j,
         v~_i  = (a_i v_i + sum_{pi(j)=i} g_j a_j v_j) / den_i          (Eq. 5)
         R_i   = den_i / a_i                                           (Eq. 6)
    with the R15 guard.  Returns (V_merged [m][d], R [m])."""
    m = kept_idx.shape[0]
    slot = {int(i): s for s, i in enumerate(kept_idx)}
    num = a_kv[kept_idx][:, None] * V_kv[kept_idx]
    den = a_kv[kept_idx].copy()
    for j in np.flatnonzero(target >= 0):
        s = slot[int(target[j])]
        w = g[j] * a_kv[j]
        num[s] += w * V_kv[j]
        den[s] += w
    Vm = np.empty_like(num)
    R = np.ones(m)
    for s in range(m):
        i = int(kept_idx[s])
        Vm[s] = num[s] / den[s] if den[s] > 0 else V_kv[i]
        if a_kv[i] > 0:
            R[s] = den[s] / a_kv[i]
    return Vm, R


def gqa_bias(R: np.ndarray, alpha: float) -> np.ndarray:
    """Sec. 3.6 for GQA: bias_i = alpha * ln(mean over KV heads of R_{kv,i}) (R16).
    R: [Hkv][m]."""
    return alpha * np.log(R.mean(axis=0))


def merge_counts(kept_idx: np.ndarray, target: np.ndarray, g: np.ndarray) -> np.ndarray:
    """M_i: the evicted tokens merged into each kept token (routed to it with g > 0), in
    kept_idx order (R19)."""
    slot = {int(i): s for s, i in enumerate(kept_idx)}
    M = np.zeros(kept_idx.shape[0])
    for j in np.flatnonzero((target >= 0) & (g > 0)):
        M[slot[int(target[j])]] += 1
    return M


def count_bias(M: np.ndarray, alpha: float, per_head: bool) -> np.ndarray:
    """R19: alpha * ln(1 + mean_kv M) (shared; M [Hkv][m] -> [m]) or alpha * ln(1 + M) per head."""
    return alpha * np.log1p(M) if per_head else alpha * np.log1p(M.mean(axis=0))


def layer_average_bias(q_layers, kept_layers, n: int, alpha: float, count: bool) -> list:
    """R21: the per-layer biases of one sequence replaced by their cross-layer average.
    q_layers[l]: layer l's per-slot quantity (KV-head mean R, or mean M in the count variant),
    shape [m] in the shared mode or [Hkv][m] per head; kept_layers[l]: the positions of those
    slots, same shape.  Returns the new bias of every layer, same shapes."""
    neutral = 0.0 if count else 1.0
    first = np.asarray(q_layers[0], dtype=np.float64)
    total = np.zeros(first.shape[:-1] + (n,))   # sum over layers, neutral where evicted
    L = len(q_layers)
    for q, kept in zip(q_layers, kept_layers):
        q = np.asarray(q, dtype=np.float64)
        kept = np.asarray(kept, dtype=np.int64)
        here = np.full(total.shape, neutral)
        np.put_along_axis(here, kept, q, axis=-1)
        total += here
    mean = total / L
    out = []
    for kept in kept_layers:
        mk = np.take_along_axis(mean, np.asarray(kept, dtype=np.int64), axis=-1)
        out.append(alpha * (np.log1p(mk) if count else np.log(mk)))
    return out


def per_head_bias(R: np.ndarray, alpha: float) -> np.ndarray:
    """Sec. 3.6 with per-head selection: bias_{h,i} = alpha * ln R_{h,i}, no averaging across
    heads (R17).  R: [Hkv][m]; returns [Hkv][m]."""
    return alpha * np.log(R)


# ----------------------------------------------------------------------------------------
# Algorithm 1 for one sequence of one layer
# ----------------------------------------------------------------------------------------
@dataclass
class CompressResult:
    m: int
    m_s: int
    a: np.ndarray             # [Hkv][n] cumulative attention
    vnorm: np.ndarray         # [Hkv][n]
    c: np.ndarray             # [Hkv][n] contribution score (Eq. 1)
    c_pooled: np.ndarray      # [Hkv][n_cand]
    sel: Optional[Selection]  # shared mode only
    kept_idx: np.ndarray      # [m] ascending (shared mode) or [Hkv][m] (per-head mode)
    target: np.ndarray        # [Hkv][n]
    g: np.ndarray             # [Hkv][n]
    sim: np.ndarray           # [Hkv][n]
    decision: np.ndarray      # [Hkv][n] uint8 (valid where target >= 0 or policy dropped)
    K_c: np.ndarray           # [Hkv][m][d]
    V_c: np.ndarray           # [Hkv][m][d]
    R: np.ndarray             # [Hkv][m]
    bias: np.ndarray          # [m] (shared mode) or [Hkv][m] (per-head mode)
    per_head: bool = False
    extra: dict = field(default_factory=dict)


def compress(K: np.ndarray, V: np.ndarray, Q: np.ndarray, n: int, rho: float,
             params: Params = Params(), follow_per_kv=None, follow_kept=None,
             follow_target=None) -> CompressResult:
    """Compression of one sequence of one layer (Sec. 3.1-3.7; RoPE repositioning, Eq. 7,
    only when params.rope is set).  K, V: [Hkv][>=n][d]; Q: [Hq][W][d]; all float64.

    follow_* replace a discrete choice of the oracle by a given one (per-KV-head top-k
    masks, final kept mask, merge targets), so that a test can compare the continuous
    outputs downstream of a near-tie the two sides resolved differently."""
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Q = np.asarray(Q, dtype=np.float64)
    Hkv = K.shape[0]
    m, m_s = budget(n, rho, params.recent)
    if m_s < 0 or Q.shape[1] > n:
        raise ValueError("budget below the recent window, or window longer than the sequence")
    n_cand = n - params.recent
    a = cumulative_attention(Q, K, n)                         # Sec. 3.1 re-pass, Eq. 1 attention sum
    vn = value_norms(V, n)
    c = a * vn                                                # Eq. 1
    cp = pool_scores(c, n_cand, params.pool_kernel)           # smoothing
    if params.select_mode == SELECT_PER_HEAD:
        return _compress_per_head(K, V, n, m, m_s, a, vn, c, cp, params, follow_per_kv, follow_target)
    sel = select_shared(cp, n, m_s, params.recent, follow_per_kv, follow_kept)  # Eq. 2, Sec. 3.3 union and trim
    kept_idx = np.flatnonzero(sel.kept)
    target = np.full((Hkv, n), -1, dtype=np.int64)
    g = np.zeros((Hkv, n))
    sim = np.zeros((Hkv, n))
    decision = np.zeros((Hkv, n), dtype=np.uint8)
    Vc = np.empty((Hkv, kept_idx.size, K.shape[2]))
    R = np.ones((Hkv, kept_idx.size))
    for kv in range(Hkv):
        t = (np.asarray(follow_target[kv][:n], dtype=np.int64) if follow_target is not None
             else _route(a[kv], V[kv], sel.kept, params))                      # Eq. 3 (Sec. 3.4)
        target[kv] = t
        g[kv], sim[kv], decision[kv] = gate(V[kv, :n], t, params.gate_mode)     # Eq. 4
        Vc[kv], R[kv] = merge(a[kv], V[kv, :n], kept_idx, t, g[kv])            # Eq. 5, Eq. 6
    if params.bias_mode == BIAS_COUNT:
        bias = count_bias(np.stack([merge_counts(kept_idx, target[kv], g[kv]) for kv in range(Hkv)]),
                          params.alpha, per_head=False)
    else:
        bias = gqa_bias(R, params.alpha)
    Kc = K[:, kept_idx].copy()
    if params.rope != ROPE_OFF:                                         # Eq. 7 (Sec. 3.7)
        Kc = np.stack([reposition(Kc[kv], kept_idx, params.rope_theta, params.rope) for kv in range(Hkv)])
    return CompressResult(m=m, m_s=m_s, a=a, vnorm=vn, c=c, c_pooled=cp, sel=sel,
                          kept_idx=kept_idx, target=target, g=g, sim=sim, decision=decision,
                          K_c=Kc, V_c=Vc, R=R, bias=bias)


def _route(a_kv, V_kv, kept, params):
    """Merge targets under the routing of params (Eq. 3 buckets, or R20 cosine; Sec. 3.4)."""
    if params.routing == ROUTE_COSINE:
        return route_cosine(V_kv, kept)
    return route(a_kv, kept, params.bucket, params.empty_bucket)


def _compress_per_head(K, V, n, m, m_s, a, vn, c, cp, params, follow_per_kv, follow_target):
    """Eq. 2-6 with per-head selection (R17; Sec. 3.3, Sec. 3.6): every KV head has its own
    kept set, targets, merged values and bias row."""
    Hkv, _, d = K.shape
    kept = select_per_head(cp, n, m_s, params.recent, follow_per_kv)      # Eq. 2 per head (Sec. 3.3)
    kept_idx = np.stack([np.flatnonzero(kept[kv]) for kv in range(Hkv)])  # [Hkv][m]
    target = np.full((Hkv, n), -1, dtype=np.int64)
    g = np.zeros((Hkv, n))
    sim = np.zeros((Hkv, n))
    decision = np.zeros((Hkv, n), dtype=np.uint8)
    Kc = np.empty((Hkv, m, d))
    Vc = np.empty((Hkv, m, d))
    R = np.ones((Hkv, m))
    for kv in range(Hkv):
        t = (np.asarray(follow_target[kv][:n], dtype=np.int64) if follow_target is not None
             else _route(a[kv], V[kv], kept[kv], params))                      # Eq. 3 (Sec. 3.4)
        target[kv] = t
        g[kv], sim[kv], decision[kv] = gate(V[kv, :n], t, params.gate_mode)     # Eq. 4
        Vc[kv], R[kv] = merge(a[kv], V[kv, :n], kept_idx[kv], t, g[kv])        # Eq. 5, Eq. 6
        Kc[kv] = K[kv, kept_idx[kv]]
        if params.rope != ROPE_OFF:                                     # Eq. 7 (Sec. 3.7)
            Kc[kv] = reposition(Kc[kv], kept_idx[kv], params.rope_theta, params.rope)
    return CompressResult(m=m, m_s=m_s, a=a, vnorm=vn, c=c, c_pooled=cp, sel=None,
                          kept_idx=kept_idx, target=target, g=g, sim=sim, decision=decision,
                          K_c=Kc, V_c=Vc, R=R,
                          bias=(count_bias(np.stack([merge_counts(kept_idx[kv], target[kv], g[kv])
                                                     for kv in range(Hkv)]), params.alpha, per_head=True)
                                if params.bias_mode == BIAS_COUNT else per_head_bias(R, params.alpha)),
                          per_head=True,
                          extra={"kept": kept})


# ----------------------------------------------------------------------------------------
# Eq. 7: RoPE repositioning
# ----------------------------------------------------------------------------------------
def rope_pairs(d: int, layout: int):
    """Index pairs (x_f, y_f) rotated together by frequency f (R18)."""
    f = np.arange(d // 2)
    if layout == ROPE_HALF:
        return f, f + d // 2
    if layout == ROPE_INTERLEAVED:
        return 2 * f, 2 * f + 1
    raise ValueError("unknown RoPE layout")


def rope(k: np.ndarray, pos: float, theta: float, layout: int) -> np.ndarray:
    """RoPE(k, pos): rotate each pair of k ([..., d]) by pos * theta^(-2f/d)."""
    k = np.asarray(k, dtype=np.float64)
    d = k.shape[-1]
    xi, yi = rope_pairs(d, layout)
    ang = pos * theta ** (-2.0 * np.arange(d // 2) / d)
    c, s = np.cos(ang), np.sin(ang)
    out = k.copy()
    out[..., xi] = k[..., xi] * c - k[..., yi] * s
    out[..., yi] = k[..., xi] * s + k[..., yi] * c
    return out


def rope_inverse(k: np.ndarray, pos: float, theta: float, layout: int) -> np.ndarray:
    """RoPE^{-1}(k, pos): the rotation by -pos * theta^(-2f/d)."""
    return rope(k, -pos, theta, layout)


def reposition(K_kept: np.ndarray, p_old: np.ndarray, theta: float, layout: int) -> np.ndarray:
    """Eq. 7: k~_s = RoPE(RoPE^{-1}(k_s, p_old[s]), s) for the kept keys in slot order."""
    out = np.empty_like(np.asarray(K_kept, dtype=np.float64))
    for s_, (k, p) in enumerate(zip(K_kept, p_old)):
        out[s_] = rope(rope_inverse(k, float(p), theta, layout), float(s_), theta, layout)
    return out


# ----------------------------------------------------------------------------------------
# Decode with the compensated cache (Alg. 1, last step; Sec. 3.6)
# ----------------------------------------------------------------------------------------
def decode(q: np.ndarray, K_c: np.ndarray, V_c: np.ndarray, bias: Optional[np.ndarray],
           length: int) -> np.ndarray:
    """out[h] = sum_{i < length} softmax_i(q_h . k_{kv(h),i} / sqrt(d) + bias_{kv(h),i}) v_i.

    q: [Hq][d]; K_c, V_c: [Hkv][>=length][d]; bias: None, [>=length] (shared by every head)
    or [Hkv][>=length].  Returns [Hq][d] float64."""
    q = np.asarray(q, dtype=np.float64)
    Hq, d = q.shape
    Hkv = K_c.shape[0]
    G = Hq // Hkv
    out = np.zeros((Hq, d))
    for h in range(Hq):
        kv = h // G
        s = (np.asarray(K_c[kv, :length], dtype=np.float64) @ q[h]) / math.sqrt(d)
        if bias is not None:
            b = np.asarray(bias, dtype=np.float64)
            s = s + (b[kv, :length] if b.ndim == 2 else b[:length])
        s = s - s.max()
        p = np.exp(s)
        p /= p.sum()
        out[h] = p @ np.asarray(V_c[kv, :length], dtype=np.float64)
    return out
