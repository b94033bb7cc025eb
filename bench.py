#!/usr/bin/env python
"""Decode-attention benchmark over DynaCalKV latent caches on GB300.

One step = one pass of the whole hot path over one decode batch:
  1. latent append of the batch's new tokens (x [B, D] . [A_k | A_v] written
     to each sequence's last cache row), then
  2. decode attention (key reconstruction on tensor cores, RoPE, online
     softmax, value absorption, split merge and B_v projection)
for every layer of the workload.  Default workload: the Llama-2-7B-like MHA
layer (D 4096, 32 heads of 128, 8 uneven key groups, sum r_g = 1024,
r_v = 1024) at batch 16 x 4096-token contexts, bf16 latents.

Metric: decode tokens/s (B queries per step), plus latent-cache GB/s and the
fraction of the HBM roofline of the main attention kernel.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config C] [--impl dck|reference]

With N > 1 (torchrun), every rank runs its own copy of the workload (the
path shards by sequence with no exchange): weak scaling, value = all ranks'
tokens / max-over-ranks time.  `--impl reference` times the fp64 CPU oracle
(the only baseline that exists: the paper has no decode kernel).
"""

from __future__ import annotations

import argparse
import hashlib
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

METRIC = "decode attn tokens/s and latent-cache HBM GB/s (% of roofline) vs context length"
UNIT = "tokens/s"
L2_FLUSH_BYTES = 512 << 20
NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e nominal, reported beside the measured copy bandwidth


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            m = json.load(f)
        return {"hbm_gbs": m["hbm_gbs"], "bf16_tflops": m["bf16_tflops"],
                "bf16_tflops_sustained": m.get("bf16_tflops_sustained", m["bf16_tflops"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def kernel_source_sha():
    """Hash of the attention kernels' code: comments and blank lines left out, so that a
    comment edit does not retire DRAM counters taken on the same code."""
    import re
    h = hashlib.sha256()
    for fn in ("decode_tc.cu", "absorb_tc.cu", "combine.cu", "tc_common.cuh", "tc_host.h", "sm100.cuh",
               "decode_simt.cu", "common.cuh"):
        p = os.path.join(ROOT, "paper_2607_24331_gb300", "csrc", fn)
        if os.path.exists(p):
            txt = open(p).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            txt = re.sub(r"//[^\n]*", "", txt)
            lines = [ln.rstrip() for ln in txt.splitlines() if ln.strip()]
            h.update("\n".join(lines).encode())
    return h.hexdigest()[:16]


def profiled_traffic(cfg):
    """DRAM bytes of one whole decode-step call (every kernel of it) from the committed ncu summary,
    if it was taken on the current kernel sources (their hash is stored beside the bytes)."""
    p = os.path.join(ROOT, "profiles", "decode_main_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(str(cfg))
    if not e or e.get("source_sha") != kernel_source_sha():
        return None
    return e.get("bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def gpu_identifier(torch, dev):
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return str(dev)


def workload_config(w, world: int) -> dict:
    """The `config` of a bench line, the same for the GPU arm and the reference arm."""
    ctx = (sorted(int(x) for x in set(w.seq_lens))[:4] if w.n_layers == 1
           else f"ragged U[1024,16384], mean {sum(w.seq_lens) / len(w.seq_lens):.0f}")
    return {"workload": w.name, "batch": w.batch, "context": ctx, "layers": w.n_layers,
            "step": "latent append of B tokens + decode attention, per layer (one dck_decode_step call)",
            "l2": "flushed between steps (512 MB write outside the timed events)",
            "parallelism": f"replicas x{world}"}


# ---------------------------------------------------------------------------
# the oracle as CPU baseline (rank 0 only)
# ---------------------------------------------------------------------------

def oracle_sample_seconds(w, budget_s, min_pairs=2, max_pairs=4096):
    """Times the fp64 oracle on (sequence, head) pairs of layer 0 until `budget_s` elapse.
    Returns (pairs, seconds, description)."""
    import numpy as np
    import oracle
    from paper_2607_24331_gb300 import synth as S

    spec = w.layer
    starts = S.seq_starts(w.seq_lens)
    q = S.gaussian(S.stream_key(w.seed, 0, S.TID["q"]), (w.batch, spec.n_q_heads, spec.head_dim), 1.0, spec.dtype)
    Bk, Bv = S.make_bk(spec, w.seed, 0), S.make_bv(spec, w.seed, 0)
    rng = np.random.default_rng(0)
    pairs, secs, cache = 0, 0.0, {}
    while (secs < budget_s or pairs < min_pairs) and pairs < max_pairs:
        b = int(rng.integers(w.batch))
        j = int(rng.integers(spec.n_q_heads))
        if b not in cache:
            L = w.seq_lens[b]
            cache = {b: (S.cache_rows(spec, w.seed, 0, "kcache", int(starts[b]), L),
                         S.cache_rows(spec, w.seed, 0, "vcache", int(starts[b]), L))}
        kc, vc = cache[b]
        t0 = time.perf_counter()
        oracle.decode_attention(spec, q[b:b + 1], kc, vc, Bk, Bv, np.array([0]), np.array([w.seq_lens[b]]),
                                heads=[j])
        secs += time.perf_counter() - t0
        pairs += 1
    desc = (f"{pairs} (sequence, query-head) pairs of layer 0 over their full contexts, fp64 numpy "
            f"(BLAS threads = host cores); tokens/s = pairs / Hq / seconds")
    return pairs, secs, desc


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(w, budget_s=12.0, config=None, batch=None):
    pairs, secs, desc = oracle_sample_seconds(w, budget_s)
    tok_s = (pairs / w.layer.n_q_heads) / secs / w.n_layers
    out = {"value": tok_s, "unit": UNIT, "cores": host_cores(), "kind": "oracle", "sample": desc}
    if config is not None:
        one = oracle_one_core(config, batch, max(1.0, budget_s / 4))
        if one:
            out["single_core"] = one
    return out


def oracle_one_core(config, batch, budget_s):
    """The same oracle timing on one host core: a child process pinned to one CPU with its BLAS and
    OpenMP pools at one thread (the pools size themselves at import, hence the separate process)."""
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
        env[k] = "1"
    cmd = [sys.executable, os.path.abspath(__file__), "--oracle-one-core", "--config", str(config),
           "--cpu-budget", str(budget_s)] + (["--batch", str(batch)] if batch else [])
    try:
        cpu = sorted(os.sched_getaffinity(0))[0]
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=max(60.0, 8 * budget_s),
                           preexec_fn=lambda: os.sched_setaffinity(0, {cpu}))
        return json.loads(r.stdout.strip().splitlines()[-1]) if r.returncode == 0 else None
    except Exception:
        return None


def run_oracle_one_core(args):
    """Child side of oracle_one_core: prints {"value", "unit", "cores", "sample"}."""
    from paper_2607_24331_gb300 import synth as S
    w = S.workload(args.config, args.batch)
    pairs, secs, desc = oracle_sample_seconds(w, args.cpu_budget)
    cores = host_cores()
    print(json.dumps({"value": (pairs / w.layer.n_q_heads) / secs / w.n_layers, "unit": UNIT, "cores": cores,
                      "sample": desc.replace("BLAS threads = host cores", "one core, BLAS threads = 1")}), flush=True)


def run_reference(args):
    from paper_2607_24331_gb300 import synth as S
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = S.workload(args.config, args.batch)
    for _ in range(args.warmup):
        oracle_sample_seconds(w, 0.0, min_pairs=1, max_pairs=1)
    t_steps, tot_pairs = [], 0
    for _ in range(args.steps):
        pairs, secs, desc = oracle_sample_seconds(w, 0.0, min_pairs=2, max_pairs=2)
        t_steps.append(secs)
        tot_pairs += pairs
    secs = sum(t_steps)
    value = (tot_pairs / w.layer.n_q_heads) / secs / w.n_layers
    line = {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, args.gpus),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": host_cores(), "kind": "oracle",
                             "sample": f"each step: 2 (sequence, query-head) pairs over full contexts, fp64 numpy"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# whole-job numbers over ranks (weak scaling: every rank runs its own replica)
# ---------------------------------------------------------------------------

def rank_seed(seed: int, rank: int) -> int:
    """Data seed of a rank's replica: each rank decodes its own sequences."""
    return seed + rank * 1000


def max_over_ranks(x: float, world: int, device) -> float:
    """The slowest rank's time: the job finishes when its last rank does."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, batch: int, steps: int, t_ms: float) -> float:
    """Decode tokens per second of the whole job: every rank decodes `batch` queries per step."""
    return world * batch * steps / (t_ms / 1e3)


# ---------------------------------------------------------------------------
# per-kernel breakdown of one decode call
# ---------------------------------------------------------------------------

def decode_kernel_names(dck, step_fn):
    """Kernels of one decode step call, in launch order (from the launch count of a plain step)."""
    step_fn()
    n = dck.dck_last_launch_count()
    if n == 4:
        return ["factor_prep+append", "scores", "absorb", "combine"]
    if n == 2:
        return ["decode_simt", "combine"]
    if n >= 3:
        return ["append"] * (n - 2) + ["decode_simt", "combine"]
    return [f"kernel{i}" for i in range(n)]


def kernel_work(buf, name):
    """Algorithmic bytes and tensor flops of one kernel of a decode call."""
    s = buf.spec
    el = 2 if s.dtype == "bf16" else 4
    d = s.head_dim
    key_flops = buf.n_rows * 2 * sum(r * len(g) for g, r in zip(s.groups, s.ranks)) * d
    val_flops = buf.n_rows * 2 * s.n_q_heads * s.rank_v
    bk = s.bk_offsets()[-1] * el
    bv = s.rank_v * s.n_kv_heads * d * el
    qo = buf.B * s.n_q_heads * d * el
    if name == "scores":
        return buf.n_rows * s.rank_k * el + bk + qo, key_flops
    if name == "absorb":
        return buf.n_rows * s.rank_v * el, val_flops
    if name == "combine":
        return bv + qo, 0
    if name == "factor_prep+append":
        app = s.hidden * (s.rank_k + s.rank_v) * el + buf.B * (s.hidden + s.rank_k + s.rank_v) * el
        return bk + qo + app, 2 * buf.B * s.hidden * (s.rank_k + s.rank_v)
    if name == "decode_simt":
        return buf.n_rows * (s.rank_k + s.rank_v) * el + bk + qo, 0
    return 0, 0


def kernel_breakdown(dck, torch, stream, flush, buf, step_fn, names, peaks, K):
    """Each kernel of the last layer's decode call timed between hook events recorded after every
    launch (a separate capture: events between kernels stop a kernel from starting early under
    programmatic dependent launch, so these sum to a little more than the call's own time)."""
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)]
    for e_ in evs:
        e_.record(stream)
    torch.cuda.synchronize()
    dck.check(dck.dck_set_timing_events(evs), "timing events")
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step_fn()
    dck.check(dck.dck_set_timing_events(None), "timing events")
    per = [[] for _ in names]
    for k in range(max(K, 3) + 2):
        flush.fill_(k & 0xFF)
        g.replay()
        torch.cuda.synchronize()
        if k >= 2:
            for i in range(len(names)):
                per[i].append(evs[i].elapsed_time(evs[i + 1]))
    out = []
    for i, n in enumerate(names):
        us = 1e3 * statistics.median(per[i])
        by, fl = kernel_work(buf, n)
        ent = {"kernel": n, "us": us, "alg_bytes": by, "tensor_flops": fl,
               "hbm_frac": by / (us * 1e-6) / 1e9 / peaks["hbm_gbs"] if us > 0 else None,
               "tensor_frac": fl / (us * 1e-6) / 1e12 / peaks["bf16_tflops"] if us > 0 else None}
        out.append(ent)
    return out


# ---------------------------------------------------------------------------
# --sweep: the measurement matrix (decode vs context length, the 32-layer step
# vs batch, every workload's call, the long-context prefill append)
# ---------------------------------------------------------------------------

def time_decode_steps(w, steps, warmup, dev, flush):
    """Decode steps (one dck_decode_step per layer) of workload w, as a CUDA graph replayed with
    L2 flushed between steps; CUDA-event times of the step and of the last layer's call."""
    import torch
    from paper_2607_24331_gb300 import dck, device
    from paper_2607_24331_gb300 import synth as S
    spec = w.layer
    B = w.batch
    dt = device.TORCH_DTYPE[spec.dtype]
    layers = []
    for l in range(w.n_layers):
        buf = device.DecodeBuffers(spec, w.seq_lens, device=dev).synth(seed=w.seed, layer=l)
        A_k = torch.empty((spec.hidden, spec.rank_k), dtype=dt, device=dev)
        A_v = torch.empty((spec.hidden, spec.rank_v), dtype=dt, device=dev)
        device.synth_fill(A_k, S.stream_key(w.seed, l, S.TID["A_k"]), 1.0 / math.sqrt(spec.hidden))
        device.synth_fill(A_v, S.stream_key(w.seed, l, S.TID["A_v"]), 1.0 / math.sqrt(spec.hidden))
        x = torch.empty((B, spec.hidden), dtype=dt, device=dev)
        device.synth_fill(x, S.stream_key(w.seed, l, S.TID["x_step"]), 1.0)
        rows = (buf.seq_start + buf.seq_len.to(torch.int64) - 1).contiguous()
        ws_s = dck.dck_decode_step_workspace_size(buf.layer, B, buf.n_rows)
        wss = torch.empty(max(ws_s, 256), dtype=torch.uint8, device=dev)
        layers.append((buf, A_k, A_v, x, rows, wss, ws_s))
    stream = torch.cuda.current_stream(dev)

    def step():
        st = torch.cuda.current_stream(dev)  # the capture stream while a graph is captured
        for buf, A_k, A_v, x, rows, wss, ws_s in layers:
            dck.check(dck.dck_decode_step(buf.layer, x, A_k, A_v, rows, buf.q, buf.kcache, buf.vcache, buf.n_rows,
                                          buf.B_k, buf.B_v, buf.seq_start, buf.seq_len, B, spec.rope_theta,
                                          buf.out, wss, ws_s, st), "decode step")

    for _ in range(warmup):
        flush.fill_(1)
        step()
    torch.cuda.synchronize()
    assert dck.dck_last_device_error(stream) == dck.DCK_OK
    kev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    for e_ in kev:
        e_.record(stream)
    torch.cuda.synchronize()
    dck.check(dck.dck_set_timing_events(kev), "timing events")
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    dck.check(dck.dck_set_timing_events(None), "timing events")
    graph.replay()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    call_ms = []
    for k in range(steps):
        flush.fill_(k & 0xFF)
        ev[k][0].record(stream)
        graph.replay()
        ev[k][1].record(stream)
        ev[k][1].synchronize()
        call_ms.append(kev[0].elapsed_time(kev[1]))
    step_ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    call_ms = statistics.median(call_ms)
    buf0 = layers[-1][0]
    el = 2 if spec.dtype == "bf16" else 4
    app_bytes = (spec.hidden * (spec.rank_k + spec.rank_v) + B * (spec.hidden + spec.rank_k + spec.rank_v)) * el
    call_bytes = buf0.algorithmic_bytes() + app_bytes
    call_flops = buf0.tensor_flops() + 2 * B * spec.hidden * (spec.rank_k + spec.rank_v)
    del graph, layers
    torch.cuda.empty_cache()
    return step_ms, call_ms, call_bytes, call_flops


def time_prefill_append(w, steps, warmup, dev, flush):
    """Latent append of w.append_tokens new tokens per sequence (dck_latent_append, rows at the end of
    each sequence), CUDA events around each call, L2 flushed between calls."""
    import numpy as np
    import torch
    from paper_2607_24331_gb300 import dck, device
    from paper_2607_24331_gb300 import synth as S
    spec = w.layer
    dt = device.TORCH_DTYPE[spec.dtype]
    n_tok = w.append_tokens * w.batch
    n_rows = sum(w.seq_lens)
    starts = S.seq_starts(w.seq_lens)
    rows_h = np.concatenate([np.arange(int(st) + L - w.append_tokens, int(st) + L) for st, L in zip(starts, w.seq_lens)])
    rows = torch.from_numpy(rows_h.astype(np.int64)).to(dev)
    x = torch.empty((n_tok, spec.hidden), dtype=dt, device=dev)
    A_k = torch.empty((spec.hidden, spec.rank_k), dtype=dt, device=dev)
    A_v = torch.empty((spec.hidden, spec.rank_v), dtype=dt, device=dev)
    kc = torch.empty((n_rows, spec.rank_k), dtype=dt, device=dev)
    vc = torch.empty((n_rows, spec.rank_v), dtype=dt, device=dev)
    device.synth_fill(x, S.stream_key(w.seed, 0, S.TID["x"]), 1.0)
    device.synth_fill(A_k, S.stream_key(w.seed, 0, S.TID["A_k"]), 1.0 / math.sqrt(spec.hidden))
    device.synth_fill(A_v, S.stream_key(w.seed, 0, S.TID["A_v"]), 1.0 / math.sqrt(spec.hidden))
    L = dck.Layer.from_spec(spec)
    wsb = dck.dck_latent_append_workspace_size(L, n_tok)
    ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def call():
        dck.check(dck.dck_latent_append(L, x, n_tok, A_k, A_v, rows, kc, vc, n_rows, ws, wsb, stream), "append")

    for _ in range(warmup):
        flush.fill_(1)
        call()
    torch.cuda.synchronize()
    assert dck.dck_last_device_error(stream) == dck.DCK_OK
    ms = []
    for k in range(steps):
        flush.fill_(k & 0xFF)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        call()
        e1.record(stream)
        e1.synchronize()
        ms.append(e0.elapsed_time(e1))
    el = 2
    bytes_ = (n_tok * spec.hidden + spec.hidden * (spec.rank_k + spec.rank_v) + n_tok * (spec.rank_k + spec.rank_v)) * el
    flops = 2 * n_tok * spec.hidden * (spec.rank_k + spec.rank_v)
    del x, kc, vc
    torch.cuda.empty_cache()
    return statistics.median(ms), bytes_, flops


def time_prefill_attention(spec, B, L, steps, warmup, dev, flush, seed=0):
    """Prefill attention (dck_prefill_attention) of B sequences whose whole L-token prompt is new
    (Q = L): CUDA events around each call, L2 flushed between calls.  Returns the median ms, the
    algorithmic bytes and the tensor flops of one call."""
    import torch
    from paper_2607_24331_gb300 import dck, device
    from paper_2607_24331_gb300 import synth as S
    dt = device.TORCH_DTYPE[spec.dtype]
    buf = device.DecodeBuffers(spec, (L,) * B, device=dev).synth(seed=seed)
    q = torch.empty((B, L, spec.n_q_heads, spec.head_dim), dtype=dt, device=dev)
    device.synth_fill(q, S.stream_key(seed, 0, S.TID["q_prefill"]), 1.0)
    ql = torch.full((B,), L, dtype=torch.int32, device=dev)
    out = torch.empty_like(q)
    wsb = dck.dck_prefill_workspace_size(buf.layer, buf.n_rows)
    ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def call():
        dck.check(dck.dck_prefill_attention(buf.layer, q, ql, L, buf.kcache, buf.vcache, buf.n_rows, buf.B_k,
                                            buf.B_v, buf.seq_start, buf.seq_len, B, L, spec.rope_theta, out, ws,
                                            wsb, stream), "prefill attention")

    for _ in range(warmup):
        flush.fill_(1)
        call()
    torch.cuda.synchronize()
    assert dck.dck_last_device_error(stream) == dck.DCK_OK
    ms = []
    for k in range(steps):
        flush.fill_(k & 0xFF)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        call()
        e1.record(stream)
        e1.synchronize()
        ms.append(e0.elapsed_time(e1))
    d, el = spec.head_dim, 2
    n = B * L
    recon = 2 * n * d * (sum(r * len(g) for g, r in zip(spec.groups, spec.ranks)) + spec.rank_v * spec.n_kv_heads)
    pairs = B * L * (L + 1) // 2                      # causal (query, key) pairs per head
    attn = 2 * 2 * pairs * d * spec.n_q_heads          # S = Q K^T and O = P V
    bytes_ = (n * (spec.rank_k + spec.rank_v) + spec.bk_offsets()[-1] + spec.rank_v * spec.n_kv_heads * d
              + 2 * n * spec.n_q_heads * d) * el
    del buf, q, out, ws
    torch.cuda.empty_cache()
    return statistics.median(ms), bytes_, recon + attn


def run_sweep(args):
    import torch
    from paper_2607_24331_gb300 import synth as S
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    peaks = load_peaks()
    steps, warmup = max(args.steps, 3), max(args.warmup, 3)
    out = {"sweep": [], "peaks": peaks}

    def line(kind, w, step_ms, call_ms, bytes_, flops, extra=None):
        ctx = sum(w.seq_lens)
        d = {"kind": kind, "workload": w.name, "batch": w.batch, "layers": w.n_layers,
             "mean_context": ctx / max(1, w.batch), "ms_per_step": step_ms, "call_us": 1e3 * call_ms,
             "decode_tokens_per_s": w.batch / (step_ms / 1e3),
             "context_tokens_per_s": ctx * w.n_layers / (step_ms / 1e3),
             "call_alg_gbs": bytes_ / (call_ms / 1e3) / 1e9,
             "hbm_frac_of_measured": bytes_ / (call_ms / 1e3) / 1e9 / peaks["hbm_gbs"],
             "tensor_frac_of_measured": flops / (call_ms / 1e3) / 1e12 / peaks["bf16_tflops"],
             "roofline_call_us": 1e6 * max(bytes_ / (peaks["hbm_gbs"] * 1e9), flops / (peaks["bf16_tflops"] * 1e12))}
        if extra:
            d.update(extra)
        out["sweep"].append(d)
        print(json.dumps(d), file=sys.stderr, flush=True)

    base = S.workload(1)
    for T in (1024, 4096, 16384, 65536):   # decode vs context length on the 7B MHA layer, B16
        w = S.Workload(f"llama2-7b-mha B16 T{T}", base.layer, (T,) * 16)
        line("context", w, *time_decode_steps(w, steps, warmup, dev, flush))
    for cfg in (0, 2, 3, 5):
        w = S.workload(cfg)
        line("workload", w, *time_decode_steps(w, steps, warmup, dev, flush))
    for b in (1, 8, 32, 64):               # the 32-layer step vs batch
        w = S.workload(4, b)
        line("32-layer step", w, *time_decode_steps(w, 3, 3, dev, flush))
    for cfg, B, L in ((1, 2, 4096), (2, 1, 8192), (3, 1, 8192)):   # prefill attention, whole prompt new
        spec = S.workload(cfg).layer
        ms, by, fl = time_prefill_attention(spec, B, L, steps, warmup, dev, flush)
        name = S.workload(cfg).name.split(" B")[0]
        out["sweep"].append({"kind": "prefill attention", "workload": f"{name}: prefill of B{B} x {L} new tokens",
                             "us": 1e3 * ms, "prompt_tokens_per_s": B * L / (ms / 1e3),
                             "tensor_tflops": fl / (ms / 1e3) / 1e12,
                             "tensor_frac_of_measured": fl / (ms / 1e3) / 1e12 / peaks["bf16_tflops"],
                             "roofline_us": 1e6 * max(by / (peaks["hbm_gbs"] * 1e9), fl / (peaks["bf16_tflops"] * 1e12))})
        print(json.dumps(out["sweep"][-1]), file=sys.stderr, flush=True)
    w3 = S.workload(3)
    ms, by, fl = time_prefill_append(w3, steps, warmup, dev, flush)
    out["sweep"].append({"kind": "prefill append", "workload": f"{w3.name}: latent append of 2 x {w3.append_tokens} tokens",
                         "us": 1e3 * ms, "tensor_tflops": fl / (ms / 1e3) / 1e12,
                         "tensor_frac_of_measured": fl / (ms / 1e3) / 1e12 / peaks["bf16_tflops"],
                         "roofline_us": 1e6 * max(by / (peaks["hbm_gbs"] * 1e9), fl / (peaks["bf16_tflops"] * 1e12))})
    print(json.dumps(out), flush=True)


# ---------------------------------------------------------------------------
# --calls: a plain driver for profilers (no timing, no JSON line)
# ---------------------------------------------------------------------------

def run_calls(args):
    """N decode-step calls (latent append + decode attention) of the first layer of the workload, L2
    flushed before each, then a check of the device error word.  ncu captures in profiles/ use it with
    `-s` to skip the first calls' kernels."""
    import torch
    from paper_2607_24331_gb300 import dck, device
    from paper_2607_24331_gb300 import synth as S
    dev = torch.device("cuda", 0)
    w = S.workload(args.config, args.batch)
    spec = w.layer
    B = w.batch
    dt = device.TORCH_DTYPE[spec.dtype]
    buf = device.DecodeBuffers(spec, w.seq_lens, device=dev).synth(seed=w.seed, layer=0)
    A_k = torch.empty((spec.hidden, spec.rank_k), dtype=dt, device=dev)
    A_v = torch.empty((spec.hidden, spec.rank_v), dtype=dt, device=dev)
    device.synth_fill(A_k, S.stream_key(w.seed, 0, S.TID["A_k"]), 1.0 / math.sqrt(spec.hidden))
    device.synth_fill(A_v, S.stream_key(w.seed, 0, S.TID["A_v"]), 1.0 / math.sqrt(spec.hidden))
    x = torch.empty((B, spec.hidden), dtype=dt, device=dev)
    device.synth_fill(x, S.stream_key(w.seed, 0, S.TID["x_step"]), 1.0)
    rows = (buf.seq_start + buf.seq_len.to(torch.int64) - 1).contiguous()
    ws_s = dck.dck_decode_step_workspace_size(buf.layer, B, buf.n_rows)
    wss = torch.empty(max(ws_s, 256), dtype=torch.uint8, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for _ in range(args.calls):
        flush.fill_(1)
        dck.check(dck.dck_decode_step(buf.layer, x, A_k, A_v, rows, buf.q, buf.kcache, buf.vcache, buf.n_rows,
                                      buf.B_k, buf.B_v, buf.seq_start, buf.seq_len, B, spec.rope_theta, buf.out,
                                      wss, ws_s), "decode step")
    torch.cuda.synchronize()
    if dck.dck_last_device_error() != dck.DCK_OK:
        raise SystemExit("device error word set")
    print(f"{args.calls} decode-step calls of {w.name}: ok", flush=True)


def run_append_calls(args):
    """N latent appends of the long-context GQA layer's prefill (2 x 8192 tokens), L2 flushed before
    each, then a check of the device error word.  The ncu capture of the append kernel in profiles/
    uses it with `-s` to skip the first calls."""
    import torch
    from paper_2607_24331_gb300 import dck
    from paper_2607_24331_gb300 import synth as S
    dev = torch.device("cuda", 0)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    w = S.workload(3)
    time_prefill_append(w, args.append_calls, 0, dev, flush)
    torch.cuda.synchronize()
    if dck.dck_last_device_error() != dck.DCK_OK:
        raise SystemExit("device error word set")
    print(f"{args.append_calls} latent appends of {w.name} (2 x {w.append_tokens} tokens): ok", flush=True)


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", type=int, default=1,
                    help="0 tiny fp32, 1 MHA B16xT4096 (default), 2/3 GQA, 4 32-layer step, 5 MHA with fixed groups of 4")
    ap.add_argument("--batch", type=int, default=None, help="batch of the 32-layer workload (config 4)")
    ap.add_argument("--impl", default="dck", choices=["dck", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--sweep", action="store_true",
                    help="measurement matrix (context lengths, workloads, 32-layer batch sweep, prefill append)")
    ap.add_argument("--oracle-one-core", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--calls", type=int, default=0,
                    help="profiling driver: this many plain decode-step calls, no timing and no JSON line")
    ap.add_argument("--append-calls", type=int, default=0,
                    help="profiling driver: this many latent appends of the long-context GQA prefill (2 x 8192 "
                         "tokens), L2 flushed before each, no JSON line")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.oracle_one_core:
        run_oracle_one_core(args)
        return
    if args.calls > 0:
        run_calls(args)
        return
    if args.append_calls > 0:
        run_append_calls(args)
        return

    if args.impl == "reference":
        run_reference(args)
        return
    if args.sweep:
        run_sweep(args)
        return

    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2607_24331_gb300 import dck, device
    from paper_2607_24331_gb300 import synth as S

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    w = S.workload(args.config, args.batch)
    spec = w.layer
    B = w.batch
    dt = device.TORCH_DTYPE[spec.dtype]
    layers = []
    for l in range(w.n_layers):
        buf = device.DecodeBuffers(spec, w.seq_lens, device=dev).synth(seed=rank_seed(w.seed, rank), layer=l)
        A_k = torch.empty((spec.hidden, spec.rank_k), dtype=dt, device=dev)
        A_v = torch.empty((spec.hidden, spec.rank_v), dtype=dt, device=dev)
        device.synth_fill(A_k, S.stream_key(w.seed, l, S.TID["A_k"]), 1.0 / math.sqrt(spec.hidden))
        device.synth_fill(A_v, S.stream_key(w.seed, l, S.TID["A_v"]), 1.0 / math.sqrt(spec.hidden))
        x = torch.empty((B, spec.hidden), dtype=dt, device=dev)
        device.synth_fill(x, S.stream_key(w.seed, l, S.TID["x_step"]), 1.0)
        rows = (buf.seq_start + buf.seq_len.to(torch.int64) - 1).contiguous()
        ws_s = dck.dck_decode_step_workspace_size(buf.layer, B, buf.n_rows)
        wss = torch.empty(max(ws_s, 256), dtype=torch.uint8, device=dev)
        layers.append((buf, A_k, A_v, x, rows, wss, ws_s))
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    launches = [0]

    def step(q_src=None, x_src=None, st=None):
        """One decode step per layer: latent append of the batch's new tokens and decode
        attention over the caches that now hold them, one dck_decode_step call."""
        st = torch.cuda.current_stream(dev) if st is None else st
        for l, (buf, A_k, A_v, x, rows, wss, ws_s) in enumerate(layers):
            xx = x if x_src is None else x_src[l]
            qq = buf.q if q_src is None else q_src[l]
            dck.check(dck.dck_decode_step(buf.layer, xx, A_k, A_v, rows, qq, buf.kcache, buf.vcache, buf.n_rows,
                                          buf.B_k, buf.B_v, buf.seq_start, buf.seq_len, B, spec.rope_theta,
                                          buf.out, wss, ws_s, st), "decode step")
            launches[0] += dck.dck_last_launch_count()

    for _ in range(args.warmup):
        flush.fill_(1)
        step()
    torch.cuda.synchronize()
    assert dck.dck_last_device_error(stream) == dck.DCK_OK

    # ---- device-resident timed region: the step is captured once as a CUDA graph;
    # two hook events bracket each decode call (every kernel of it) ----
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    kev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    for e_ in kev:               # torch creates the CUDA event on first record
        e_.record(stream)
    torch.cuda.synchronize()
    dck.check(dck.dck_set_timing_events(list(kev)), "timing events")
    graph = torch.cuda.CUDAGraph()
    launches[0] = 0
    with torch.cuda.graph(graph):
        step()
    per_step_launches = launches[0]
    dck.check(dck.dck_set_timing_events(None), "timing events")
    decode_kernels = decode_kernel_names(dck, step)
    for _ in range(args.warmup):
        flush.fill_(1)
        graph.replay()
    torch.cuda.synchronize()
    clocks = ClockSampler(gpu_identifier(torch, local))
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    kern_ms = []
    for k in range(K):
        flush.fill_(k & 0xFF)
        ev[k][0].record(stream)
        graph.replay()
        ev[k][1].record(stream)
        ev[k][1].synchronize()
        kern_ms.append(kev[0].elapsed_time(kev[1]))
    torch.cuda.synchronize()
    # the same steps with L2 left warm (reported beside the flushed headline)
    wev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    for k in range(K):
        wev[k][0].record(stream)
        graph.replay()
        wev[k][1].record(stream)
    torch.cuda.synchronize()
    warm_ms = statistics.median(a.elapsed_time(b) for a, b in wev)
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    launches[0] = per_step_launches * K
    gpu_launches = launches[0]
    step_ms = [a.elapsed_time(b) for a, b in ev]
    t_ms = max_over_ranks(sum(step_ms), world, dev)
    ms_per_step = t_ms / K
    value = job_throughput(world, B, K, t_ms)

    # ---- end to end: host inputs -> device -> result back, every step ----
    q_host = [torch.empty(buf.q.shape, dtype=dt, pin_memory=True) for (buf, *_r) in layers]
    x_host = [torch.empty(x.shape, dtype=dt, pin_memory=True) for (_b, _a, _v, x, *_r) in layers]
    out_host = [torch.empty(buf.out.shape, dtype=dt, pin_memory=True) for (buf, *_r) in layers]
    for l, (buf, _a, _v, x, *_r) in enumerate(layers):
        q_host[l].copy_(buf.q)
        x_host[l].copy_(x)
    q_dev = [torch.empty_like(buf.q) for (buf, *_r) in layers]
    x_dev = [torch.empty_like(x) for (_b, _a, _v, x, *_r) in layers]
    h2d = sum(t.numel() * t.element_size() for t in q_host + x_host)
    d2h = sum(t.numel() * t.element_size() for t in out_host)

    def e2e_step():
        for l in range(len(layers)):
            q_dev[l].copy_(q_host[l], non_blocking=True)
            x_dev[l].copy_(x_host[l], non_blocking=True)
        step(q_dev, x_dev)
        for l, (buf, *_r) in enumerate(layers):
            out_host[l].copy_(buf.out, non_blocking=True)

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    eev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    if world > 1:
        dist.barrier()
    for k in range(K):
        flush.fill_(k & 0xFF)
        eev[k][0].record(stream)
        e2e_step()
        eev[k][1].record(stream)
        eev[k][1].synchronize()   # the result is on the host before the next step starts
    e2e_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in eev), world, dev)
    e2e_value = job_throughput(world, B, K, e2e_ms)

    # ---- roofline of one whole decode-step call (append + decode attention: every kernel
    # between the two hook events; one call = one layer), then a per-kernel breakdown ----
    peaks = load_peaks()
    buf0 = layers[-1][0]
    el0 = 2 if spec.dtype == "bf16" else 4
    app_bytes = (spec.hidden * (spec.rank_k + spec.rank_v) + B * (spec.hidden + spec.rank_k + spec.rank_v)) * el0
    alg_bytes = buf0.algorithmic_bytes() + app_bytes
    flops = buf0.tensor_flops() + 2 * B * spec.hidden * (spec.rank_k + spec.rank_v)
    k_avg_s = statistics.mean(kern_ms) / 1e3
    achieved_gbs = alg_bytes / k_avg_s / 1e9
    tflops = flops / k_avg_s / 1e12
    step_alg_bytes = len(layers) * alg_bytes
    roof = {"bound": "hbm", "achieved": achieved_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved_gbs / peaks["hbm_gbs"], "traffic": profiled_traffic(args.config),
            "kernel": "one whole decode-step call: " + " + ".join(decode_kernels), "kernel_us": 1e6 * k_avg_s,
            "alg_bytes_per_launch": alg_bytes, "peak_source": peaks["source"],
            "tensor_tflops": tflops, "tensor_frac": tflops / peaks["bf16_tflops"],
            "roofline_us": 1e6 * max(alg_bytes / (peaks["hbm_gbs"] * 1e9), flops / (peaks["bf16_tflops"] * 1e12)),
            "frac_of_nominal_8000gbs": achieved_gbs / NOMINAL_HBM_GBS,
            "breakdown": kernel_breakdown(dck, torch, stream, flush, buf0, step, decode_kernels, peaks, K)}

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": args.warmup,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if spec.dtype == "bf16" else "f32", "data": "synthetic (seeded Gaussian latents/factors)",
            "config": workload_config(w, world),
            "latent_gbs": step_alg_bytes / (ms_per_step / 1e3) / 1e9,
            "context_tokens_per_s": world * sum(w.seq_lens) * w.n_layers / (ms_per_step / 1e3),
            "ms_per_step_median": statistics.median(step_ms), "ms_per_step_warm_l2": warm_ms,
            "roofline": roof, "clocks": clk,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": gpu_launches}
    if rank == 0 and world == 1:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_budget, args.config, args.batch)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
