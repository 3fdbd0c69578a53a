"""SelKV benchmark: one-shot compression of a 32-layer GQA cache followed by compensated
decode, on synthetic inputs of the paper's latency setting (Llama-3-8B attention shape,
100k-token context, 25% budget, 256 generated tokens).

One step = compress every layer (selkv_compress) + decode_steps tokens, each token running
selkv_decode_attn on every layer with a fresh query and an appended key/value row.
`value` = generated tokens / step time (compression included); the decode-only rate,
compress ms per layer, decode GB/s and the roofline of the decode kernel are reported beside
it.  Inputs are resident in HBM when the timed region starts; `e2e` repeats the step through
the public API from pinned host buffers with the copies inside the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload long_100k]
  python bench.py --impl reference ...    (the fp64 CPU oracle on a bounded sample)
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "compensated decode tokens/s & HBM GB/s (% peak) at 100k ctx; compress ms/layer"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(PEAKS_FALLBACK), "fallback"


# ------------------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ------------------------------------------------------------------------------ oracle arm
def _oracle_unit(job):
    """One unit of the oracle baseline: generate layer `layer` of sequence 0, compress it with
    the fp64 oracle, then decode `tokens` tokens over the compressed cache (each appending a
    row).  Returns the times and the process's CPU time."""
    wl, layer, tokens, per_head = job
    from oracle import selkv_oracle as O
    cpu0 = time.process_time()
    one = wl.with_(batch=1)
    x = synth.gen_layer(one, layer, threads=1)
    n = int(x["n_len"][0])
    K, V, Q = (x[k][0].astype(np.float64) for k in ("K", "V", "Q_obs"))
    t0 = time.perf_counter()
    r = O.compress(K, V, Q, n, wl.rho, O.Params(select_mode=O.SELECT_PER_HEAD if per_head else O.SELECT_SHARED))
    t_comp = time.perf_counter() - t0
    dec = synth.gen_decode(one, layer, tokens)
    Kc, Vc, bias = r.K_c, r.V_c, r.bias
    t_dec = 0.0
    for t in range(tokens):
        Kc = np.concatenate([Kc, dec["k_new"][t, 0][:, None]], axis=1)
        Vc = np.concatenate([Vc, dec["v_new"][t, 0][:, None]], axis=1)
        bias = np.concatenate([bias, np.zeros(bias.shape[:-1] + (1,))], axis=-1)
        t0 = time.perf_counter()
        O.decode(dec["q"][t, 0], Kc, Vc, bias, Kc.shape[1])
        t_dec += time.perf_counter() - t0
    return {"compress_s": t_comp, "decode_s_per_token": t_dec / max(1, tokens),
            "cpu_s": time.process_time() - cpu0}


def _blas_threads_env(threads: int):
    """Environment for worker processes: `threads` BLAS / OpenMP threads each."""
    keys = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS")
    old = {k: os.environ.get(k) for k in keys}
    for k in keys:
        os.environ[k] = str(threads)
    return old


def _restore_env(old):
    for k, v in old.items():
        if v is None:
            os.environ.pop(k, None)
        else:
            os.environ[k] = v


class _OraclePool:
    """P spawned worker processes with `blas_threads` BLAS threads each; spawned, not forked,
    so that no worker inherits a CUDA context."""

    def __init__(self, P: int, blas_threads: int = 1):
        self.P = P
        self.blas_threads = blas_threads

    @classmethod
    def for_step(cls, wl):
        """As many workers as the step has (sequence, layer) units, at most one per core, and
        the cores shared out among them as BLAS threads (one each when the units outnumber the
        cores; all of them for a one-unit step)."""
        cores = os.cpu_count() or 1
        P = max(1, min(cores, wl.batch * wl.layers))
        return cls(P, max(1, cores // P))

    def __enter__(self):
        import multiprocessing as mp
        old = _blas_threads_env(self.blas_threads)
        try:
            self.pool = mp.get_context("spawn").Pool(self.P)
        finally:
            _restore_env(old)
        return self

    def __exit__(self, *exc):
        self.pool.terminate()
        self.pool.join()

    def units(self, wl, first_layer: int, tokens: int, per_head: bool):
        """P units at once: worker i compresses layer (first_layer + i) mod L of sequence 0 and
        decodes `tokens` tokens over it.  Returns the units' results and the wall time."""
        jobs = [(wl, (first_layer + i) % wl.layers, tokens, per_head) for i in range(self.P)]
        t0 = time.perf_counter()
        res = self.pool.map(_oracle_unit, jobs, chunksize=1)
        return res, time.perf_counter() - t0


def _step_rate(wl, res, P: int):
    """Tokens per second of the workload's step from a sample of (sequence, layer) units run P
    at once: the step's B x L units take ceil(B L / P) rounds of the mean unit (compression +
    decode_steps decode tokens).  Returns (rate, rounds)."""
    unit_s = statistics.mean(r["compress_s"] + wl.decode_steps * r["decode_s_per_token"] for r in res)
    rounds = math.ceil(wl.batch * wl.layers / P)
    return wl.batch * wl.decode_steps / (rounds * unit_s), rounds


def oracle_sample(wl: synth.Workload, per_head: bool = False, decode_tokens: int = 2,
                  single_thread_refs: bool = True) -> dict:
    """The fp64 oracle on the host's cores, parallel over independent units: one spawned worker
    process per (sequence, layer) unit of the step up to one per core (single-threaded BLAS
    when the units outnumber the cores, the cores shared out as BLAS threads otherwise), each
    compressing one layer of sequence 0 (layers 0 .. P-1) and decoding `decode_tokens` tokens
    over it; all P run at once, so each unit's time is taken under the memory contention of a
    full machine.  The step estimate schedules the step's B x L units on the P workers:
    ceil(B L / P) rounds of the mean unit time (compression + decode_steps decode tokens).
    With single_thread_refs, the tiny and the 16k single-layer workloads are also timed alone
    on one core each (compression and decode per layer)."""
    refs = [(synth.WORKLOADS["tiny"], 0, 16, False), (synth.WORKLOADS["llama_layer"], 0, 2, False)]
    with _OraclePool.for_step(wl) as pool:
        res, wall = pool.units(wl, 0, decode_tokens, per_head)
    P, threads = pool.P, pool.blas_threads
    single = None
    if single_thread_refs:
        with _OraclePool(len(refs), 1) as rp:
            single = rp.pool.map(_oracle_unit, refs, chunksize=1)
    value, rounds = _step_rate(wl, res, P)
    busy = sum(r["cpu_s"] for r in res) / wall
    out = {"value": value, "unit": "tokens/s", "cores": P * threads, "kind": "oracle",
           "sample": ("fp64 oracle, %d worker process(es) (%d BLAS thread(s) each) at once, "
                      "each compressing one layer of one sequence (n=%d) and decoding %d token(s); "
                      "the step's %d (sequence, layer) units scheduled as %d round(s) of the mean "
                      "unit (compression + %d decode tokens)")
           % (P, threads, wl.n, decode_tokens, wl.batch * wl.layers, rounds, wl.decode_steps),
           "compress_s_per_layer": statistics.mean(r["compress_s"] for r in res),
           "decode_s_per_layer_token": statistics.mean(r["decode_s_per_token"] for r in res),
           "sample_wall_s": wall, "cores_busy_avg": round(busy, 2)}
    if single is not None:
        out["single_thread"] = {
            w.name: {"compress_s": r["compress_s"], "decode_s_per_token": r["decode_s_per_token"],
                     "tokens_per_s": w.decode_steps / (w.layers * (r["compress_s"]
                                                                   + w.decode_steps * r["decode_s_per_token"]))}
            for (w, _, _, _), r in zip(refs, single)}
    return out


# ------------------------------------------------------------------------------ ranks
def max_over_ranks(x: float, torch, dist, device) -> float:
    """The largest x over all ranks (x itself without a process group of several ranks):
    the job's time is that of its slowest rank."""
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() < 2:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def decode_bytes_per_launch(wl, n_len, T: int, per_head: bool = False) -> float:
    """Algorithmic bytes of one decode launch (one layer, one token), averaged over T tokens:
    each cached row of each KV head reads its K_c and V_c rows (d elements each), and each
    cached position its fp32 bias (one value per position shared by the KV heads in the shared
    selection mode, one per KV head in the per-head mode), the row appended at step t included
    (a sequence holds m_b + t + 1 rows at step t); plus the queries and outputs of every query
    head and the appended key and value rows.  (The kernel reads the shared-mode bias from
    every KV head's copy of the row: 4 (Hkv - 1) bytes per position more than counted here.)"""
    esz = 2 if wl.dtype == "bf16" else 4
    d, Hkv, Hq = wl.head_dim, wl.num_kv_heads, wl.num_q_heads
    m_b = [int(math.floor(wl.rho * n)) for n in n_len]
    per_row = Hkv * 2 * d * esz + 4 * (Hkv if per_head else 1)
    rows_total = sum(sum(m + t + 1 for t in range(T)) for m in m_b)   # over the T steps
    fixed = T * len(n_len) * (2 * Hq * d * esz + 2 * Hkv * d * esz)
    return (rows_total * per_row + fixed) / T


def whole_job_rate(world: int, units_per_rank: float, seconds: float) -> float:
    """Units processed by all ranks per second (weak scaling: every rank does the same work)."""
    return world * units_per_rank / seconds


# ------------------------------------------------------------------------------ GPU arm
class HostArena:
    """Page-locked host memory for the end-to-end inputs: one allocation from the CUDA
    runtime (cudaHostAlloc through torch), carved into the host copies of the inputs.  On a
    GB300 (Grace host, NVLink-C2C) it streams to the device at ~210 GB/s when copies run back
    to back; a region of 512 MiB transparent huge pages registered with cudaHostRegister
    measured no faster in the end-to-end loop (and depends on the kernel finding the huge
    pages)."""

    def __init__(self, torch, nbytes: int):
        self.torch = torch
        self.total = (nbytes + 255) // 256 * 256
        self.base = torch.empty(self.total, dtype=torch.uint8, pin_memory=True)
        self.off = 0

    def take(self, like):
        """A page-locked host copy of `like`."""
        n = like.numel() * like.element_size()
        assert self.off + n <= self.total
        t = self.base[self.off:self.off + n].view(like.dtype).view(like.shape)
        self.off += (n + 255) // 256 * 256
        t.copy_(like)
        return t


class Layered:
    """Device-resident inputs and outputs of every layer."""

    def __init__(self, wl, torch, api, S, dev, pinned_host: bool, layer_average: bool = False,
                 compress_streams: int = 1):
        self.wl = wl
        self.torch = torch
        B, Hq, Hkv, d, W = wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.obs_window
        tdt = api.torch_dtype(api.dtype_code(wl.dtype))
        self.n_len = [int(v) for v in synth.seq_lengths(wl)]
        self.T = wl.decode_steps
        self.m_cap = api.capacity(max(self.n_len), wl.rho, extra=self.T + 1)
        self.shape = api.make_shape(wl.dtype, B, Hq, Hkv, d, W, wl.n, self.m_cap)
        self.K, self.V, self.Q, self.caches, self.host = [], [], [], [], []
        self.arena = None
        if pinned_host:
            es = 2 if wl.dtype == "bf16" else 4
            per_layer = (2 * B * Hkv * wl.n * d + B * Hq * W * d) * es + 3 * 256
            # every token's q, k_new, v_new and every token's outputs
            decode = wl.decode_steps * wl.layers * B * (2 * Hq + 2 * Hkv) * d * es + 4 * 256
            self.arena = HostArena(torch, wl.layers * per_layer + decode)
        threads = os.cpu_count() or 1
        for layer in range(wl.layers):
            x = synth.gen_layer(wl, layer, threads=threads)
            K = torch.from_numpy(x["K"]).to(dev).to(tdt)
            V = torch.from_numpy(x["V"]).to(dev).to(tdt)
            Q = torch.from_numpy(x["Q_obs"]).to(dev).to(tdt)
            self.K.append(K)
            self.V.append(V)
            self.Q.append(Q)
            if pinned_host:
                self.host.append(tuple(self.arena.take(t) for t in (K, V, Q)))
            self.caches.append(api.alloc_compressed(self.shape, dev))
        # decode inputs for every (step, layer): q [T][L][B][Hq][d], k/v [T][L][B][Hkv][d]
        qs, ks, vs = [], [], []
        for layer in range(wl.layers):
            dd = synth.gen_decode(wl, layer, self.T)
            qs.append(dd["q"])
            ks.append(dd["k_new"])
            vs.append(dd["v_new"])
        self.dq = torch.from_numpy(np.stack(qs, 1)).to(dev).to(tdt)
        self.dk = torch.from_numpy(np.stack(ks, 1)).to(dev).to(tdt)
        self.dv = torch.from_numpy(np.stack(vs, 1)).to(dev).to(tdt)
        self.out = torch.empty((self.T, wl.layers, B, Hq, d), dtype=tdt, device=dev)
        self.cws = api.Workspace(S.selkv_compress_workspace_size(self.shape), dev)
        # layers are compressed on `compress_streams` streams in turn (the caller's first), each
        # with its own workspace; the extra streams fork from the caller's and join it again
        self.comp_streams = [torch.cuda.Stream(device=dev) for _ in range(max(1, compress_streams) - 1)]
        self.comp_ws = [api.Workspace(S.selkv_compress_workspace_size(self.shape), dev)
                        for _ in self.comp_streams]
        self.dws = api.Workspace(S.selkv_decode_workspace_size(self.shape), dev)
        # compensation averaged across layers: each layer's kept positions are kept for it
        self.layer_average = layer_average
        # (sized for the per-head mode's [B][Hkv][m_cap]; the shared mode uses the first B m_cap)
        self.kept = [torch.empty((B, Hkv, self.m_cap), dtype=torch.int32, device=dev) for _ in range(wl.layers)] \
            if layer_average else []
        self.aws = api.Workspace(S.selkv_layer_average_workspace_size(self.shape), dev) if layer_average else None


def compress_layers(L: Layered, S, params, stream_ptr, before_layer=None, inputs=None):
    """Enqueue the compression of every layer (and, with layer averaging, the average) on the
    current stream (`stream_ptr`), layer l on stream l mod (1 + extra streams) with that
    stream's workspace: the compressions of a model's layers after prefill are independent, and
    the latency-bound selection kernels of one layer leave room for another layer's work.
    `inputs` = (K, V, Q) lists of device tensors per layer (default: the resident ones);
    `before_layer(layer, stream)` may make the stream that compresses the layer wait."""
    wl = L.wl
    torch = L.torch
    main = torch.cuda.current_stream()
    assert main.cuda_stream == stream_ptr, "compress_layers enqueues on the current stream"
    streams = [main] + L.comp_streams
    wss = [L.cws] + L.comp_ws
    Ks, Vs, Qs = inputs if inputs is not None else (L.K, L.V, L.Q)
    for st in L.comp_streams:
        st.wait_stream(main)
    for layer in range(wl.layers):
        k = layer % len(streams)
        if before_layer is not None:
            before_layer(layer, streams[k])
        c = L.caches[layer]
        dbg = {"kept_idx": L.kept[layer]} if L.layer_average else None
        S.check(S.selkv_compress(L.shape, L.n_len, wl.rho, params, Ks[layer], Vs[layer], Qs[layer],
                                 c.K_c, c.V_c, c.bias, c.lengths, dbg, wss[k].buf, wss[k].nbytes,
                                 streams[k].cuda_stream), "compress")
    for st in L.comp_streams:
        main.wait_stream(st)
    if L.layer_average:
        S.check(S.selkv_layer_average_bias(L.shape, params, L.kept, [c.bias for c in L.caches],
                                           L.caches[0].lengths, L.aws.buf, L.aws.nbytes, stream_ptr),
                "layer average")


def issue_step(L: Layered, S, params, stream_ptr, decode_ranges=None):
    """Enqueue one step on the stream; returns the number of kernels enqueued."""
    wl = L.wl
    k0 = S.selkv_kernel_launches()
    compress_layers(L, S, params, stream_ptr)
    if decode_ranges is not None:
        decode_ranges[0]()
    for t in range(L.T):
        for layer in range(wl.layers):
            c = L.caches[layer]
            S.check(S.selkv_decode_attn(L.shape, L.dq[t, layer], c.K_c, c.V_c, c.bias, c.lengths,
                                        L.dk[t, layer], L.dv[t, layer], L.out[t, layer],
                                        L.dws.buf, L.dws.nbytes, stream_ptr), "decode")
    return S.selkv_kernel_launches() - k0


def run_gpu(args):
    import torch
    import torch.distributed as dist
    import paper_2607_16213_gb300 as S
    from paper_2607_16213_gb300 import api, build as _build

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    _build.build()
    S.library()
    wl = synth.WORKLOADS[args.workload]
    if args.decode_steps is not None:
        wl = wl.with_(decode_steps=args.decode_steps)
    if args.layers is not None:
        wl = wl.with_(layers=args.layers)
    params = S.selkv_params.defaults(
        select_mode=S.SELKV_SELECT_PER_HEAD if args.select_mode == "per_head" else S.SELKV_SELECT_SHARED,
        rope={"off": S.SELKV_ROPE_OFF, "half": S.SELKV_ROPE_HALF,
              "interleaved": S.SELKV_ROPE_INTERLEAVED}[args.rope], rope_theta=args.rope_theta,
        routing=S.SELKV_ROUTE_COSINE if args.routing == "cosine" else S.SELKV_ROUTE_BUCKET)
    L = Layered(wl, torch, api, S, dev, pinned_host=not args.no_e2e, layer_average=args.layer_average,
                compress_streams=args.compress_streams)
    # inputs, caches and workspaces were initialised on the default stream; the work below runs
    # on other streams, which do not wait for it
    torch.cuda.synchronize()
    stream = torch.cuda.Stream(device=dev)
    sp = stream.cuda_stream
    peaks, peak_src = load_peaks()

    with torch.cuda.stream(stream):
        launches_per_step = issue_step(L, S, params, sp)   # one eager step (also warms up)
    torch.cuda.synchronize()
    assert L.cws.errors(sp) == 0 and L.dws.errors(sp) == 0, "device error flags"

    # capture compression and decode as two graphs, so the timed region is launch-free
    g_comp = torch.cuda.CUDAGraph()
    g_dec = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_comp, stream=stream):
        compress_layers(L, S, params, stream.cuda_stream)
    with torch.cuda.graph(g_dec, stream=stream):
        for t in range(L.T):
            for layer in range(wl.layers):
                c = L.caches[layer]
                S.check(S.selkv_decode_attn(L.shape, L.dq[t, layer], c.K_c, c.V_c, c.bias, c.lengths,
                                            L.dk[t, layer], L.dv[t, layer], L.out[t, layer],
                                            L.dws.buf, L.dws.nbytes, stream.cuda_stream), "decode")
    n_dec_launch = L.T * wl.layers
    for _ in range(args.warmup):
        g_comp.replay()
        g_dec.replay()
    torch.cuda.synchronize()

    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    clocks = ClockSampler(torch.cuda.current_device() if not os.environ.get("CUDA_VISIBLE_DEVICES") else 0)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    # one more untimed step: the clocks ramp down while the sampler starts
    with torch.cuda.stream(stream):
        g_comp.replay()
        g_dec.replay()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    with torch.cuda.stream(stream):
        for k in range(args.steps):
            ev[k][0].record(stream)
            g_comp.replay()
            ev[k][1].record(stream)
            g_dec.replay()
            ev[k][2].record(stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t_wall
    clk = clocks.stop()
    # every replayed step must have left the caches where one eager step leaves them: each
    # layer's lengths at m_b + T (compression resets them, each token appends one row), and no
    # device error flag raised
    want = [int(math.floor(wl.rho * n)) + L.T for n in L.n_len]
    for layer, c in enumerate(L.caches):
        got = c.lengths.cpu().tolist()
        assert got == want, "layer %d lengths %s after the timed steps, expected %s" % (layer, got[:4], want[:4])
    assert L.cws.errors(sp) == 0 and L.dws.errors(sp) == 0, "device error flags after the timed steps"
    comp_ms = [ev[k][0].elapsed_time(ev[k][1]) for k in range(args.steps)]
    dec_ms = [ev[k][1].elapsed_time(ev[k][2]) for k in range(args.steps)]
    step_ms_total = max_over_ranks(ev[0][0].elapsed_time(ev[-1][2]), torch, dist, dev)
    if world > 1:
        dist.barrier()
    ms_per_step = step_ms_total / args.steps
    tokens_per_step = wl.batch * L.T
    value = whole_job_rate(world, tokens_per_step * args.steps, step_ms_total / 1e3)
    dec_ms_avg = sum(dec_ms) / len(dec_ms)
    comp_ms_avg = sum(comp_ms) / len(comp_ms)
    decode_tok_s = tokens_per_step / (dec_ms_avg / 1e3)

    d, Hkv, Hq, B = wl.head_dim, wl.num_kv_heads, wl.num_q_heads, wl.batch
    dec_bytes_per_layer_step = decode_bytes_per_launch(wl, L.n_len, L.T, per_head=args.select_mode == "per_head")
    dec_launch_us = dec_ms_avg * 1e3 / n_dec_launch
    achieved_gbs = dec_bytes_per_layer_step / (dec_launch_us * 1e-6) / 1e9
    peak_hbm = float(peaks["hbm_gbs"])
    traffic = None
    prof = os.path.join(ROOT, "profiles", "decode_traffic.json")
    if os.path.exists(prof):
        with open(prof) as f:
            pj = json.load(f)
        if pj.get("workload") == wl.name and pj.get("kernel_rev") == kernel_revision(
                S.selkv_decode_workspace_size(L.shape)):
            traffic = pj.get("bytes_per_launch")

    score = None if args.no_score else measure_scoring(L, S, api, torch, stream, dev, peaks, peak_src)

    # full-cache comparison (same kernel, bias = NULL, uncompressed cache, no append)
    full_tok_s = None
    if not args.no_full:
        fshape = api.make_shape(wl.dtype, B, Hq, Hkv, d, wl.obs_window, wl.n, wl.n)
        flen = torch.tensor(L.n_len, dtype=torch.int32, device=dev)
        fws = api.Workspace(S.selkv_decode_workspace_size(fshape), dev)
        torch.cuda.synchronize()   # flen and fws are ready before `stream` uses them
        nfull = max(2, min(16, L.T))
        def full_pass():
            for t in range(nfull):
                for layer in range(wl.layers):
                    S.check(S.selkv_decode_attn(fshape, L.dq[t, layer], L.K[layer], L.V[layer], None, flen,
                                                None, None, L.out[t, layer], fws.buf, fws.nbytes, sp), "full")
        with torch.cuda.stream(stream):
            full_pass()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            full_pass()
            e1.record(stream)
        torch.cuda.synchronize()
        full_tok_s = B * nfull / (e0.elapsed_time(e1) / 1e3)

    # end to end through the public API from pinned host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(L, S, api, torch, params, stream, dev, args.e2e_steps, args.warmup)
        e2e["ms_per_step"] = max_over_ranks(e2e["ms_per_step"], torch, dist, dev)
        e2e["value"] = whole_job_rate(world, wl.batch * L.T, e2e["ms_per_step"] / 1e3)

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": wl.name, "layers": wl.layers, "batch": wl.batch, "n": wl.n,
                   "rho": wl.rho, "decode_steps": L.T, "q_heads": Hq, "kv_heads": Hkv,
                   "head_dim": d, "obs_window": wl.obs_window, "select_mode": args.select_mode,
                   "rope": args.rope, "routing": args.routing,
                   "compensation": "averaged across layers" if args.layer_average else "per layer",
                   "parallelism": "replicas", "compress_streams": max(1, args.compress_streams),
                   "l2": (("inputs larger than L2: every token streams all layers' compressed "
                           "caches (%.2f GB)" % (dec_bytes_per_layer_step * wl.layers / 1e9))
                          if dec_bytes_per_layer_step * wl.layers > 2 * L2_BYTES else
                          ("L2-resident: the workload's compressed caches (%.0f MB per token over all "
                           "layers) fit in L2, so the decode figures are not HBM figures"
                           % (dec_bytes_per_layer_step * wl.layers / 1e6))),
                   "cuda_graph": True},
        "decode_tok_s": decode_tok_s,
        "decode_gbs": achieved_gbs,
        "compress_ms_per_layer": comp_ms_avg / wl.layers,
        "full_cache_decode_tok_s": full_tok_s,
        "decode_speedup_vs_full_cache": (decode_tok_s / full_tok_s) if full_tok_s else None,
        "roofline": {"kernel": "selkv decode (split-K, GQA, bias in softmax)", "bound": "hbm",
                     "achieved": achieved_gbs, "peak": peak_hbm, "unit": "GB/s",
                     "frac": achieved_gbs / peak_hbm, "peak_source": peak_src,
                     "bytes_per_launch": dec_bytes_per_layer_step,
                     "launch_us": dec_launch_us, "traffic": traffic},
        "roofline_score": score,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
        "wall_s_timed": wall,
    }
    if e2e is not None:
        line["e2e"] = e2e
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.routing == "bucket" and not args.layer_average:
        line["cpu_baseline"] = oracle_sample(wl, per_head=args.select_mode == "per_head")
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def score_flops_per_pass(wl, n_len) -> float:
    """Flops of one pass of the scoring: the product of the G W window rows of every KV head
    with all n_b keys (2 d flops per score), over every sequence; the causal corner is
    computed and masked, so executed and algorithmic flops agree.  The method needs this one
    product; the second pass repeats it (it needs the row normalisers of the first)."""
    return float(sum(2.0 * wl.num_q_heads * wl.obs_window * n * wl.head_dim for n in n_len))


def measure_scoring(L: Layered, S, api, torch, stream, dev, peaks, peak_src, reps: int = 3) -> dict:
    """The scoring stage (selkv_score) of every layer, its two passes timed apart: first the
    row-statistics pass of all layers back to back (each layer its own small workspace), then
    the column-sum pass of all layers; CUDA events around each group, per-pass time = group
    time / layers (median over `reps`).  Every layer reads its own K (205 MB at 100k context),
    so nothing stays in L2 from one layer to the next."""
    wl = L.wl
    sp = stream.cuda_stream
    wss = [api.Workspace(S.selkv_score_workspace_size(L.shape), dev) for _ in range(wl.layers)]
    attn = torch.empty((wl.batch, wl.num_kv_heads, wl.n), dtype=torch.float32, device=dev)
    torch.cuda.synchronize()   # the workspaces are zeroed before `stream` uses them
    rounds = []
    with torch.cuda.stream(stream):
        for r in range(reps + 1):
            e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            e[0].record(stream)
            for layer in range(wl.layers):
                S.check(S.selkv_score(L.shape, L.n_len, L.K[layer], L.Q[layer], None, S.SELKV_SCORE_ROWSTATS,
                                      wss[layer].buf, wss[layer].nbytes, sp), "score pass 1")
            e[1].record(stream)
            for layer in range(wl.layers):
                S.check(S.selkv_score(L.shape, L.n_len, L.K[layer], L.Q[layer], attn, S.SELKV_SCORE_COLSUMS,
                                      wss[layer].buf, wss[layer].nbytes, sp), "score pass 2")
            e[2].record(stream)
            if r > 0:   # the first round warms up
                rounds.append(e)
    torch.cuda.synchronize()
    assert all(w.errors(sp) == 0 for w in wss), "device error flags in the scoring"
    p1 = statistics.median(x[0].elapsed_time(x[1]) for x in rounds) * 1e3 / wl.layers
    p2 = statistics.median(x[1].elapsed_time(x[2]) for x in rounds) * 1e3 / wl.layers
    F = score_flops_per_pass(wl, L.n_len)
    peak = float(peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"]))
    burst = float(peaks["bf16_tflops"])
    r1, r2 = F / (p1 * 1e-6) / 1e12, F / (p2 * 1e-6) / 1e12
    stage = F / ((p1 + p2) * 1e-6) / 1e12
    return {"kernel": "selkv scoring (tcgen05, two passes over K)" if wl.dtype == "bf16" else "selkv scoring",
            "bound": "tensor", "unit": "TFLOP/s", "peak": peak, "peak_burst": burst, "peak_source": peak_src,
            "flops_per_pass": F, "pass1_us": p1, "pass2_us": p2,
            "pass1_tflops": r1, "pass2_tflops": r2,
            "pass1_frac": r1 / peak, "pass2_frac": r2 / peak,
            "pass1_frac_burst": r1 / burst, "pass2_frac_burst": r2 / burst,
            "achieved": 2 * F / ((p1 + p2) * 1e-6) / 1e12, "frac": 2 * F / ((p1 + p2) * 1e-6) / 1e12 / peak,
            "useful_tflops_stage": stage, "useful_frac_stage": stage / peak,
            "note": "pass 1 includes the sequence-table upload and the fold of the row statistics; "
                    "achieved = executed flops of both passes over their time; useful = one product "
                    "(what the method needs) over the stage's time; peaks: sustained, and burst beside",
            "traffic": None}


def run_e2e(L: Layered, S, api, torch, params, stream, dev, steps: int, warmup: int):
    """The step through the public API with its inputs in pinned host memory: every layer's
    K, V and Q_obs and every token's q, k_new and v_new are copied from host to device, every
    layer is compressed, the tokens are decoded (each token every layer, appending), and every
    token's outputs are read back to host memory.  Steps are double-buffered: the input
    copies of step i + 1 (on a copy stream, into the other of two device input sets) run while
    step i computes; layer l of a step compresses once its copies have landed and the token
    loop starts once the token inputs have.  The token loop (the decode calls only) is
    captured once per input set as a CUDA graph; the compression calls are issued eagerly; the
    outputs go back on a third stream once the step's token loop is done.  Every timed step
    moves its full input and output bytes across the link inside the timed region (the input
    copies for the first timed step run during the last warm-up step; those issued during the
    last timed step, and the last outputs, are waited for before the clock stops).  The
    per-token inputs travel with the step's other inputs rather than token by token: a small
    copy queued behind the layers' bulk copies on the host link would stall its token for the
    length of the bulk transfer.  Host buffers come from a HostArena."""
    wl = L.wl
    sp = stream.cuda_stream
    hq = L.arena.take(L.dq)
    hk = L.arena.take(L.dk)
    hv = L.arena.take(L.dv)
    hout = L.arena.take(torch.empty(L.out.shape, dtype=L.out.dtype))
    h2d = sum(t.numel() * t.element_size() for trip in L.host for t in trip) + \
        sum(t.numel() * t.element_size() for t in (hq, hk, hv))
    d2h = hout.numel() * hout.element_size()

    # two device input sets: the resident one and a second of the same shapes
    sets = [(L.K, L.V, L.Q, L.dq, L.dk, L.dv),
            ([torch.empty_like(x) for x in L.K], [torch.empty_like(x) for x in L.V],
             [torch.empty_like(x) for x in L.Q], torch.empty_like(L.dq), torch.empty_like(L.dk),
             torch.empty_like(L.dv))]
    copy_stream = torch.cuda.Stream(device=dev)
    out_stream = torch.cuda.Stream(device=dev)
    arrived = [[torch.cuda.Event() for _ in range(wl.layers)] for _ in range(2)]
    tok_arrived = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]  # last kernel of a step that read the set
    decoded = torch.cuda.Event()
    torch.cuda.synchronize()

    def tokens(si):
        _, _, _, dq, dk, dv = sets[si]
        for t in range(L.T):
            for layer in range(wl.layers):
                api.decode(L.caches[layer], dq[t, layer], dk[t, layer], dv[t, layer], out=L.out[t, layer],
                           workspace=L.dws, stream=sp)

    g_tok = []
    for si in range(2):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            tokens(si)
        g_tok.append(g)
    torch.cuda.synchronize()

    copy_marks = []   # (start, end) events around each step's input copies

    def copy_inputs(si, after=None):
        """Enqueue the host-to-device copies of a step's inputs into input set si."""
        Ks, Vs, Qs, dq, dk, dv = sets[si]
        with torch.cuda.stream(copy_stream):
            if after is not None:
                copy_stream.wait_event(after)
            m0, m1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            m0.record(copy_stream)
            for layer in range(wl.layers):
                hK, hV, hQ = L.host[layer]
                Ks[layer].copy_(hK, non_blocking=True)
                Vs[layer].copy_(hV, non_blocking=True)
                Qs[layer].copy_(hQ, non_blocking=True)
                arrived[si][layer].record(copy_stream)
            dq.copy_(hq, non_blocking=True)
            dk.copy_(hk, non_blocking=True)
            dv.copy_(hv, non_blocking=True)
            tok_arrived[si].record(copy_stream)
            m1.record(copy_stream)
            copy_marks.append((m0, m1))

    def one(i):
        si = i % 2
        with torch.cuda.stream(stream):
            compress_layers(L, S, params, sp, inputs=sets[si][:3],
                            before_layer=lambda layer, st: st.wait_event(arrived[si][layer]))
            stream.wait_event(tok_arrived[si])
            stream.wait_event(decoded)     # the previous step's outputs have been read back
            g_tok[si].replay()
            consumed[si].record(stream)
        # the step's outputs go back once its tokens are decoded
        with torch.cuda.stream(out_stream):
            out_stream.wait_event(consumed[si])
            hout.copy_(L.out, non_blocking=True)
            decoded.record(out_stream)
        # the next step's inputs go to the other set once the step that last read it is done
        copy_inputs(1 - si, after=consumed[1 - si] if i > 0 else None)

    copy_inputs(0)
    for i in range(warmup):
        one(i)
    torch.cuda.synchronize()
    first = len(copy_marks)
    t0 = time.perf_counter()
    for i in range(warmup, warmup + steps):
        one(i)
    stream.synchronize()
    out_stream.synchronize()
    copy_stream.synchronize()
    dt = (time.perf_counter() - t0) / steps
    bulk = sum(t.numel() * t.element_size() for trip in L.host for t in trip) + \
        sum(t.numel() * t.element_size() for t in (hq, hk, hv))
    copy_ms = [a.elapsed_time(b) for a, b in copy_marks[first:]]
    return {"value": wl.batch * L.T / dt, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": dt * 1e3, "steps": steps, "warmup": warmup,
            "pipelined": "the next step's input copies overlap this step's compute",
            "input_copy_gbs": [round(bulk / (ms * 1e-3) / 1e9, 1) for ms in copy_ms]}


# ------------------------------------------------------------------------------ serving sweep
SWEEP_METRIC = "serving sweep point: compensated decode HBM GB/s per launch; compress ms/layer"
L2_BYTES = 126 * 2 ** 20


def parse_sweep(name: str):
    """'sweep:B,n,rho' -> (B, n, rho)."""
    b, n, r = name.split(":", 1)[1].split(",")
    return int(b), int(n), float(r)


def compress_bytes(wl, n_len) -> float:
    """Algorithmic bytes of one layer's compression: every sequence reads its K and V rows and
    its window queries once and writes its kept K_c and V_c rows and one fp32 bias per kept
    position."""
    esz = 2 if wl.dtype == "bf16" else 4
    d, Hkv, Hq, W = wl.head_dim, wl.num_kv_heads, wl.num_q_heads, wl.obs_window
    tot = 0
    for n in n_len:
        m = int(math.floor(wl.rho * n))
        tot += 2 * Hkv * n * d * esz + Hq * W * d * esz + 2 * Hkv * m * d * esz + m * 4
    return float(tot)


def oracle_sweep_sample(wl, n_len, T: int) -> dict:
    """The fp64 oracle on a bounded sample of one sweep point: compression of sequence 0 and
    one decode token over its compressed cache, scaled to the layer (every sequence, by its
    length) and to T decode tokens."""
    from oracle import selkv_oracle as O
    x = synth.gen_sequence(wl, 0, 0, threads=os.cpu_count() or 1)
    n0 = x["n"]
    K, V, Q = (x[k].astype(np.float64) for k in ("K", "V", "Q_obs"))
    t0 = time.perf_counter()
    r = O.compress(K, V, Q, n0, wl.rho)
    t_comp = time.perf_counter() - t0
    dec = synth.gen_decode(wl.with_(batch=1), 0, 1)
    t0 = time.perf_counter()
    O.decode(dec["q"][0, 0], r.K_c, r.V_c, r.bias, r.m)
    t_dec = time.perf_counter() - t0
    m0 = r.m
    comp_layer = t_comp * sum(n_len) / n0
    dec_layer = t_dec * sum(int(math.floor(wl.rho * n)) for n in n_len) / m0
    return {"value": comp_layer * 1e3, "unit": "ms/layer (compression)", "cores": os.cpu_count(),
            "kind": "oracle", "decode_ms_per_layer_token": dec_layer * 1e3,
            "sample": "fp64 oracle: compression of sequence 0 (n=%d) and one decode token over its "
                      "cache, scaled by length to the %d sequences of the layer" % (n0, len(n_len))}


def sweep_point(args, point, torch, S, api, dev, peaks, peak_src) -> dict:
    """One point of the batched serving sweep (ragged lengths, one layer): compression of the
    layer timed from a cold L2 (an L2-sized buffer is written before each timed replay), then
    decode over the compressed cache, T tokens each appending a row.  Decode runs over enough
    copies of the compressed layer (up to 32, as a 32-layer model would hold) that one token's
    caches exceed three times L2; if even 32 copies do not, the L2 is flushed before every
    token and the flush's own time (measured alone) is subtracted."""
    B, n, rho = point
    wl = synth.sweep(B, n, rho)
    T = wl.decode_steps
    Hq, Hkv, d, W = wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.obs_window
    n_len = [int(v) for v in synth.seq_lengths(wl)]
    m_cap = api.capacity(max(n_len), rho, extra=T + 1)
    shape = api.make_shape(wl.dtype, B, Hq, Hkv, d, W, n, m_cap)
    bf = torch.bfloat16
    K = torch.zeros((B, Hkv, n, d), dtype=bf, device=dev)
    V = torch.zeros((B, Hkv, n, d), dtype=bf, device=dev)
    Q = torch.empty((B, Hq, W, d), dtype=bf, device=dev)
    for b in range(B):
        x = synth.gen_sequence(wl, 0, b, threads=os.cpu_count() or 1)
        nb = x["n"]
        K[b, :, :nb].copy_(torch.from_numpy(x["K"]).to(bf))
        V[b, :, :nb].copy_(torch.from_numpy(x["V"]).to(bf))
        Q[b].copy_(torch.from_numpy(x["Q_obs"]).to(bf))
        del x
    params = S.selkv_params.defaults()
    stream = torch.cuda.Stream(device=dev)
    sp = stream.cuda_stream
    cache = api.alloc_compressed(shape, dev)
    ws = api.Workspace(S.selkv_compress_workspace_size(shape), dev)
    torch.cuda.synchronize()   # zeroed on the default stream; `stream` does not wait for it

    def compress():
        S.check(S.selkv_compress(shape, n_len, rho, params, K, V, Q, cache.K_c, cache.V_c, cache.bias,
                                 cache.lengths, None, ws.buf, ws.nbytes, sp), "compress")

    m_b = [int(math.floor(rho * v)) for v in n_len]
    with torch.cuda.stream(stream):
        compress()
    torch.cuda.synchronize()
    assert ws.errors(sp) == 0
    if cache.lengths.cpu().tolist() != m_b:
        raise RuntimeError("lengths after the first compression: %s, expected %s"
                           % (cache.lengths.cpu().tolist()[:8], m_b[:8]))
    g_comp = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_comp, stream=stream):
        compress()
    lengths0 = torch.tensor(m_b, dtype=torch.int32, device=dev)

    dec_bytes = decode_bytes_per_launch(wl, n_len, T)
    copies = max(1, min(32, int(math.ceil(3 * L2_BYTES / dec_bytes))))
    flush_tokens = copies * dec_bytes < 2 * L2_BYTES
    caches = [cache] + [api.CompressedCache(shape=shape, K_c=cache.K_c.clone(), V_c=cache.V_c.clone(),
                                            bias=cache.bias.clone(), lengths=cache.lengths.clone())
                        for _ in range(copies - 1)]
    dd = synth.gen_decode(wl, 0, T)
    dq, dk, dv = (torch.from_numpy(dd[k]).to(dev).to(bf) for k in ("q", "k_new", "v_new"))
    out = torch.empty((T, B, Hq, d), dtype=bf, device=dev)
    dws = api.Workspace(S.selkv_decode_workspace_size(shape), dev)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()   # the copies, inputs and workspace are ready before `stream` uses them
    g_dec, g_flush = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_dec, stream=stream):
        for t in range(T):
            if flush_tokens:
                flush.zero_()
            for c in caches:
                S.check(S.selkv_decode_attn(shape, dq[t], c.K_c, c.V_c, c.bias, c.lengths, dk[t], dv[t], out[t],
                                            dws.buf, dws.nbytes, sp), "decode")
    with torch.cuda.graph(g_flush, stream=stream):
        for t in range(T):
            flush.zero_()

    def reset_lengths():
        for c in caches:
            c.lengths.copy_(lengths0)

    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            flush.zero_()
            g_comp.replay()
            if i == 0:
                comp_len = cache.lengths.clone()
            reset_lengths()
            g_dec.replay()
            g_flush.replay()
    torch.cuda.synchronize()
    if comp_len.cpu().tolist() != m_b:
        raise RuntimeError("lengths after a replayed compression: %s, expected %s"
                           % (comp_len.cpu().tolist()[:8], m_b[:8]))
    steps = max(args.steps, 10)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(steps)]
    clocks = ClockSampler(torch.cuda.current_device() if not os.environ.get("CUDA_VISIBLE_DEVICES") else 0)
    clocks.start()
    time.sleep(0.3)
    with torch.cuda.stream(stream):
        for k in range(steps):
            flush.zero_()
            ev[k][0].record(stream)
            g_comp.replay()
            ev[k][1].record(stream)
            reset_lengths()
            ev[k][2].record(stream)
            g_dec.replay()
            ev[k][3].record(stream)
            if flush_tokens:
                ev[k][4].record(stream)
                g_flush.replay()
                ev[k][5].record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    want = [m + T for m in m_b]
    cflags, dflags = ws.errors(sp), dws.errors(sp)
    for i, c in enumerate(caches):
        got = c.lengths.cpu().tolist()
        if got != want:
            bad = [(b, got[b], want[b]) for b in range(B) if got[b] != want[b]]
            raise RuntimeError("lengths after the timed decode (copy %d of %d; (seq, got, want) %s; "
                               "device flags compress %#x decode %#x; m_cap %d)"
                               % (i, copies, bad[:8], cflags, dflags, m_cap))
    assert cflags == 0 and dflags == 0, "device error flags %#x %#x" % (cflags, dflags)
    comp_ms = statistics.median(ev[k][0].elapsed_time(ev[k][1]) for k in range(steps))
    dec_ms = statistics.median(ev[k][2].elapsed_time(ev[k][3]) for k in range(steps))
    flush_ms = statistics.median(ev[k][4].elapsed_time(ev[k][5]) for k in range(steps)) if flush_tokens else 0.0
    launch_us = (dec_ms - flush_ms) * 1e3 / (T * copies)
    dec_gbs = dec_bytes / (launch_us * 1e-6) / 1e9
    c_bytes = compress_bytes(wl, n_len)
    comp_gbs = c_bytes / (comp_ms * 1e-3) / 1e9
    peak_hbm = float(peaks["hbm_gbs"])
    line = {
        "metric": SWEEP_METRIC, "value": dec_gbs, "unit": "GB/s", "n_gpus": 1, "steps": steps,
        "warmup": args.warmup, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": wl.name, "batch": B, "n": n, "rho": rho, "n_len_min": min(n_len),
                   "n_len_max": max(n_len), "layers_timed": 1, "layers_reported": 32,
                   "decode_steps": T, "q_heads": Hq, "kv_heads": Hkv, "head_dim": d, "obs_window": W,
                   "decode_layer_copies": copies,
                   "l2": ("compression: L2 flushed before each timed replay; decode: %s"
                          % ("L2 flushed before each token, the flush time subtracted" if flush_tokens
                             else "one token streams %.0f MB of caches (> 3x L2)" % (copies * dec_bytes / 1e6))),
                   "cuda_graph": True},
        "compress_ms_per_layer": comp_ms,
        "compress_ms_x32": 32 * comp_ms,
        "compress_gbs": comp_gbs,
        "decode_launch_us": launch_us,
        "decode_tok_s_x32": B / (32 * launch_us * 1e-6),
        "roofline": {"kernel": "selkv decode (split-K, GQA, bias in softmax)", "bound": "hbm",
                     "achieved": dec_gbs, "peak": peak_hbm, "unit": "GB/s", "frac": dec_gbs / peak_hbm,
                     "peak_source": peak_src, "bytes_per_launch": dec_bytes, "launch_us": launch_us,
                     "traffic": None},
        "roofline_compress": {"bound": "hbm", "achieved": comp_gbs, "peak": peak_hbm, "unit": "GB/s",
                              "frac": comp_gbs / peak_hbm, "bytes_per_layer": c_bytes},
        "clocks": clk,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = oracle_sweep_sample(wl, n_len, T)
    del K, V, Q, caches, cache, ws, dws, flush, g_comp, g_dec, g_flush
    torch.cuda.empty_cache()
    return line


def run_sweep(args, points):
    import torch
    import paper_2607_16213_gb300 as S
    from paper_2607_16213_gb300 import api, build as _build
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    _build.build()
    S.library()
    peaks, peak_src = load_peaks()
    failed = 0
    for pt in points:
        try:
            line = sweep_point(args, pt, torch, S, api, dev, peaks, peak_src)
        except (RuntimeError, AssertionError) as e:   # report the point and go on with the others
            failed += 1
            line = {"metric": SWEEP_METRIC, "config": {"workload": synth.sweep(*pt).name}, "error": str(e)}
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
        print(json.dumps(line), flush=True)
    if failed:
        sys.exit(1)


DECODE_SOURCES = ("decode_tc.cu", "decode_common.cuh", "ptx.cuh", "selkv_internal.cuh", "tma_host.cu")


def kernel_revision(plan_bytes: int) -> str:
    """Content hash of the tensor-core decode kernel's sources and of its launch plan for the
    workload (the decode workspace size, which grows with the split count the host picks):
    profiler figures recorded for the decode kernel are valid only for this revision."""
    import hashlib
    h = hashlib.sha256()
    cs = os.path.join(ROOT, "paper_2607_16213_gb300", "csrc")
    for f in DECODE_SOURCES:
        with open(os.path.join(cs, f), "rb") as fh:
            h.update(fh.read())
    h.update(b"plan:%d" % int(plan_bytes))
    return h.hexdigest()[:16]


def run_reference(args):
    """The oracle arm: the fp64 oracle on the host's cores, parallel over independent units as
    in the main line's `cpu_baseline` (one spawned worker per (sequence, layer) unit up to one
    per core, the cores left over shared out as BLAS threads; the pool kept for the whole run).
    Each step is one bounded sample of the workload's step: the P workers each compress a
    different layer of sequence 0 (the next P layers every step) and decode 8 tokens over it,
    all at once; the step's B x L units are scheduled as ceil(B L / P) rounds of the mean unit.
    Warm-up steps decode one token.  The line reports the median over the steps."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1 and rank != 0:
        return
    wl = synth.WORKLOADS[args.workload]
    if args.decode_steps is not None:
        wl = wl.with_(decode_steps=args.decode_steps)
    per_head = args.select_mode == "per_head"
    tokens_per_sample = 8
    vals, comp, dec, cpu_s, walls = [], [], [], 0.0, 0.0
    with _OraclePool.for_step(wl) as pool:
        P, threads = pool.P, pool.blas_threads
        for i in range(args.warmup):
            pool.units(wl, i * P, 1, per_head)
        for k in range(args.steps):
            res, wall = pool.units(wl, (args.warmup + k) * P, tokens_per_sample, per_head)
            vals.append(_step_rate(wl, res, P)[0])
            comp.append(statistics.mean(r["compress_s"] for r in res))
            dec.append(statistics.mean(r["decode_s_per_token"] for r in res))
            cpu_s += sum(r["cpu_s"] for r in res)
            walls += wall
    v = statistics.median(vals)
    tokens = wl.batch * wl.decode_steps
    rounds = math.ceil(wl.batch * wl.layers / P)
    sample = ("fp64 oracle, %d worker process(es) (%d BLAS thread(s) each) at once: per step each "
              "compresses one layer of one sequence (n=%d; %d different layer(s) a step) and decodes "
              "%d tokens over it; the step's %d (sequence, layer) units scheduled as %d round(s) of the "
              "mean unit (compression + %d decode tokens)"
              % (P, threads, wl.n, min(P, wl.layers), tokens_per_sample, wl.batch * wl.layers, rounds,
                 wl.decode_steps))
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": tokens / v * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": wl.name, "layers": wl.layers, "batch": wl.batch, "n": wl.n,
                       "rho": wl.rho, "decode_steps": wl.decode_steps, "q_heads": wl.num_q_heads,
                       "kv_heads": wl.num_kv_heads, "head_dim": wl.head_dim, "obs_window": wl.obs_window,
                       "select_mode": args.select_mode},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": P * threads, "kind": "oracle",
                             "sample": sample, "cores_busy_avg": round(cpu_s / max(1e-9, walls), 2),
                             "compress_s_per_layer": statistics.median(comp),
                             "decode_s_per_layer_token": statistics.median(dec)},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="selkv", choices=["selkv", "reference"])
    ap.add_argument("--workload", default="long_100k",
                    help="one of %s, or sweep:B,n,rho (a point of the batched serving sweep)"
                         % ", ".join(synth.WORKLOADS))
    ap.add_argument("--sweep", default=None,
                    help="serving-sweep points, 'all' or 'B,n,rho;B,n,rho;...': one JSON line each")
    ap.add_argument("--decode-steps", type=int, default=None)
    ap.add_argument("--layers", type=int, default=None, help=argparse.SUPPRESS)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10, help="timed steps of the end-to-end measurement")
    ap.add_argument("--no-full", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-score", action="store_true", help="skip the timing of the scoring passes")
    ap.add_argument("--select-mode", default="shared", choices=["shared", "per_head"],
                    help="token selection: shared (GQA union, the default) or per_head (MHA)")
    ap.add_argument("--rope", default="off", choices=["off", "half", "interleaved"],
                    help="RoPE repositioning of the kept keys (Eq. 7; off in the paper's configuration)")
    ap.add_argument("--rope-theta", type=float, default=500000.0)
    ap.add_argument("--routing", default="bucket", choices=["bucket", "cosine"],
                    help="routing of the evicted tokens: bucket (Eq. 3, the default) or the full "
                         "cosine routing of Sec. 3.4 (the oracle baseline is not sampled for it)")
    ap.add_argument("--compress-streams", type=int, default=4,
                    help="streams the layers' compressions are spread over (each with its own workspace)")
    ap.add_argument("--layer-average", action="store_true",
                    help="compensation averaged across layers instead of per layer (Sec. 3 overview)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.sweep is not None:
        pts = synth.SWEEP_POINTS if args.sweep == "all" else [
            (int(b), int(n), float(r)) for b, n, r in (p.split(",") for p in args.sweep.split(";"))]
        run_sweep(args, pts)
    elif args.impl == "reference":
        run_reference(args)
    elif args.workload.startswith("sweep:"):
        run_sweep(args, [parse_sweep(args.workload)])
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
