"""Benchmark of one structured-suffix (SSM) denoising pass on GB300.

A bench step is one pass of the whole hot path -- suffix selection, sparse
step input with soft suffix embeddings, bidirectional attention, unmasking --
over one batch of synthetic input.  The default workload is the long-sequence
LLaDA-8B shape (32 heads, head_dim 128, 1024-token prompt in a prefix cache,
2048 generated tokens, block 32, budgets local 64 / middle 64 / tail 16) with
every block index 0..63 decoded as one batch of 64 independent denoising
steps, so one bench step = 64 denoising steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload long|serve|dream|llada|tiny]
    python bench.py --impl reference ...   # the fp64 CPU oracle on the host cores

Prints one JSON line (rank 0).  Multi-GPU runs (torchrun, one process per GPU)
are independent replicas: the path has no exchange step.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_23167_gb300 import workloads as W  # noqa: E402

METRIC = "structured-suffix attn TFLOP/s (% bf16 peak); denoise steps/s; unmask HBM GB/s"
UNIT = "denoise-steps/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_BYTES = 129 * 1000 * 1000          # GB300 L2
FLUSH_BYTES = 256 * 1024 * 1024       # written between timed steps whose inputs fit in twice the L2
SLEEP_CYCLES = 1_000_000              # GPU-side delay (~0.5 ms) ahead of each stage-timing step


# ----------------------------------------------------------------------------- workload


def suffix_positions(w: W.Workload, b: int):
    """Host-side count of R_t from the library's pure host function (no device work)."""
    from paper_2608_23167_gb300 import ssm
    nl, nm, nt = ssm.ssm_suffix_count(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
    return nl + nm + nt


class StepInputs:
    """Device-resident synthetic inputs of one bench step, plus the problem tables."""

    def __init__(self, w: W.Workload, device, seed: int = 1234):
        from paper_2608_23167_gb300 import ssm
        self.w = w
        self.dev = device
        blocks = list(w.block_indices)
        self.problems = [(s, b) for s in range(w.batch) for b in blocks]
        n = len(self.problems)
        self.n = n
        self.cfgs = [(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail) for _, b in self.problems]
        self.R = [suffix_positions(w, b) for _, b in self.problems]
        # without a prefix cache the step recomputes the prompt and the blocks already decoded
        # (one block index per batch here, so one prefix length)
        if not w.prefix_cached and len(set(blocks)) != 1:
            raise ValueError("a workload without prefix cache takes one block index per step")
        n_prefix = 0 if w.prefix_cached else w.prompt + blocks[0] * w.block
        self.n_prefix = n_prefix
        self.rows = [n_prefix + w.block + r for r in self.R]          # sparse-input rows per problem
        self.row_off = np.concatenate([[0], np.cumsum(self.rows)]).astype(np.int64)
        self.suf_off = np.concatenate([[0], np.cumsum(self.R)]).astype(np.int64)
        self.total_rows = int(self.row_off[-1])
        self.total_suffix = int(self.suf_off[-1])
        V, H, k = w.vocab, w.hidden, w.topk
        self.mask_id = V - 1
        g = torch.Generator(device=device)
        g.manual_seed(seed)
        # model state: embedding table and (for the cached configurations) the prefix cache
        self.embed = (torch.randn((V, H), generator=g, device=device) * 1.0).to(torch.bfloat16)
        if w.prefix_cached:
            if w.name == "long":
                # one sequence: every block index reads the same cache, positions [0, prompt + b*B)
                self.cache_rows = w.prompt + w.gen
                self.cache_row = [0 for _ in self.problems]
            else:
                # one cache per sequence, long enough for its largest block index's prefix
                seg = w.prompt + max(blocks) * w.block
                self.cache_rows = w.batch * seg
                self.cache_row = [s * seg for s, _ in self.problems]
            self.n_cache = [w.prompt + b * w.block for _, b in self.problems]
            self.k_cache = torch.randn((self.cache_rows, w.h_kv, w.head_dim), generator=g, device=device).to(torch.bfloat16)
            self.v_cache = torch.randn((self.cache_rows, w.h_kv, w.head_dim), generator=g, device=device).to(torch.bfloat16)
        else:
            self.cache_rows = 0
            self.cache_row = [0] * n
            self.n_cache = [0] * n
            self.k_cache = self.v_cache = None
        # per-step inputs: block tokens (first step of each block: all masked), previous-step
        # top-k candidates, projections of the sparse input (stand-ins), LM-head logits (stand-ins)
        self.block_tokens = torch.full((n, w.block), self.mask_id, dtype=torch.int32, device=device)
        self.prefix_tokens = (torch.randint(0, V - 1, (n, n_prefix), generator=g, device=device, dtype=torch.int32)
                              if n_prefix else None)
        self.topk_ids = torch.randint(0, V - 1, (max(self.total_suffix, 1), k), generator=g, device=device,
                                      dtype=torch.int32)
        z = torch.softmax(torch.randn((max(self.total_suffix, 1), k), generator=g, device=device) * 3.0, dim=1)
        self.topk_prob = (torch.sort(z, dim=1, descending=True).values *
                          (0.2 + 0.8 * torch.rand((z.shape[0], 1), generator=g, device=device))).contiguous()
        self.q = torch.randn((self.total_rows, w.h_q, w.head_dim), generator=g, device=device).to(torch.bfloat16)
        self.k = torch.randn((self.total_rows, w.h_kv, w.head_dim), generator=g, device=device).to(torch.bfloat16)
        self.v = torch.randn((self.total_rows, w.h_kv, w.head_dim), generator=g, device=device).to(torch.bfloat16)
        lg = torch.randn((n, w.block, V), generator=g, device=device) * w.logits_sigma
        self.logits = lg.to(torch.bfloat16) if w.logits_dtype == "bf16" else lg
        del lg
        self.masked = (self.block_tokens == self.mask_id).to(torch.uint8)
        # outputs and scratch
        self.positions = torch.zeros(max(self.total_suffix, 1), dtype=torch.int32, device=device)
        self.x = torch.empty((self.total_rows, H), dtype=torch.bfloat16, device=device)
        self.pos = torch.empty(self.total_rows, dtype=torch.int32, device=device)
        self.out = torch.empty_like(self.q)
        self.conf = torch.empty((n, w.block), dtype=torch.float32, device=device)
        self.argmax = torch.empty((n, w.block), dtype=torch.int32, device=device)
        self.p2 = torch.empty((n, w.block), dtype=torch.float32, device=device)
        self.commit = torch.empty((n, w.block), dtype=torch.uint8, device=device)
        self.attn_ws = torch.empty(ssm.ssm_attention_workspace_size(self.total_rows, w.h_q, w.h_kv, w.head_dim),
                                   dtype=torch.uint8, device=device)
        self.unmask_ws = torch.empty(ssm.ssm_unmask_workspace_size(n, w.block, V, self.logits.dtype),
                                     dtype=torch.uint8, device=device)
        self.step_tab = ssm.step_problems_tensor(
            [(i * w.block, i * n_prefix, int(self.suf_off[i]), int(self.row_off[i]), n_prefix, self.R[i],
              W.block_start(w, b)) for i, (_, b) in enumerate(self.problems)], device)
        self.cfg_tab = ssm.suffix_cfgs_tensor(self.cfgs, device)
        self.attn_tab = ssm.attn_problems_tensor(
            [(int(self.row_off[i]), self.cache_row[i], self.rows[i], self.n_cache[i]) for i in range(n)], device)
        self.max_rows = max(self.rows)
        self.max_cache = max(self.n_cache)

    # -- algorithmic work of one step ------------------------------------------------------
    def attn_flops(self) -> float:
        w = self.w
        return float(sum(4.0 * w.h_q * w.head_dim * r * (r + c) for r, c in zip(self.rows, self.n_cache)))

    def attn_bytes(self) -> float:
        w = self.w
        e = 2
        qo = 2 * self.total_rows * w.h_q * w.head_dim * e
        kv_new = 2 * self.total_rows * w.h_kv * w.head_dim * e
        cache = 2 * (self.cache_rows if self.k_cache is not None else 0) * w.h_kv * w.head_dim * e
        return float(qo + kv_new + cache)

    def rope_bytes(self) -> float:
        """Algorithmic bytes of the RoPE pre-pass: new query and key rows read once, written rotated."""
        w = self.w
        return float(2 * self.total_rows * (w.h_q + w.h_kv) * w.head_dim * 2)

    def gather_rows_read(self) -> int:
        """Distinct embedding rows one launch of the gather reads: the [MASK] row once, plus the
        distinct ids among the prompt, block and previous-step top-k tokens (a row read twice in
        one launch is served by the L2 the second time, so it is counted once)."""
        if getattr(self, "_rows_read", None) is None:
            ids = [self.block_tokens.flatten(), self.topk_ids[:self.total_suffix].flatten(),
                   torch.tensor([self.mask_id], dtype=torch.int32, device=self.dev)]
            if self.prefix_tokens is not None:
                ids.append(self.prefix_tokens.flatten())
            allids = torch.cat(ids)
            self._rows_read = int(torch.unique(allids[allids >= 0]).numel())
        return self._rows_read

    def gather_rows_read_gross(self) -> int:
        """Embedding row reads one launch issues, repeats included."""
        w = self.w
        return sum(self.n_prefix + w.block + w.topk * r for r in self.R) + 1

    def gather_bytes(self) -> float:
        """Algorithmic bytes of the gather: distinct embedding rows read once, output rows written."""
        return float((self.gather_rows_read() + self.total_rows) * self.w.hidden * 2)

    def step_bytes(self) -> float:
        """Algorithmic bytes one step reads and writes (gather, attention, unmasking)."""
        return self.gather_bytes() + self.attn_bytes() + self.unmask_bytes()

    def unmask_bytes(self) -> float:
        w = self.w
        masked_rows = int(self.masked.sum())
        return float(masked_rows * w.vocab * self.logits.element_size())

    # -- one pass of the hot path ---------------------------------------------------------
    def step(self, ev=None, unmask=None):
        from paper_2608_23167_gb300 import ssm
        w = self.w
        if ev is not None:
            ev[0].record()
            ev[1].record()   # selection is made inside the gather launch: its own stage is empty
        # selection (Eqs. 1-5) and the sparse input (Eqs. 6-8) in one launch
        ssm.ssm_select_build_step_input_varlen(self.step_tab, self.cfg_tab, self.n, self.max_rows, w.block,
                                               self.block_tokens, self.embed, self.mask_id, self.topk_ids,
                                               self.topk_prob, w.topk, w.alpha, self.x, self.pos, self.positions,
                                               prefix_tokens=self.prefix_tokens)
        if ev is not None:
            ev[2].record()
        # the attention stage as its two launches (RoPE pre-pass, forward), timed apart
        args = (self.q, self.k, self.v, self.pos, self.k_cache, self.v_cache, self.attn_tab, self.n,
                self.max_rows, self.max_cache, self.out, w.rope_theta)
        ssm.ssm_attention_varlen_rotate(*args, workspace=self.attn_ws)
        if ev is not None:
            ev[3].record()
        ssm.ssm_attention_varlen_core(*args, workspace=self.attn_ws)
        if ev is not None:
            ev[4].record()
        # the threshold rule needs no second-largest probability, so p2 is not requested
        if unmask is not None:
            unmask()
        else:
            ssm.ssm_unmask(self.logits, self.masked, self.conf, self.argmax, self.commit, p2=None,
                           threshold=w.threshold, min_commit=1, workspace=self.unmask_ws)
        if ev is not None:
            ev[5].record()

    LAUNCHES_PER_STEP = 5   # select + build, rope_pack, attn_fwd, unmask stream, unmask commit

    def attn_core(self):
        """The attention forward alone on the step's rotated inputs (the step has run once)."""
        from paper_2608_23167_gb300 import ssm
        w = self.w
        ssm.ssm_attention_varlen_core(self.q, self.k, self.v, self.pos, self.k_cache, self.v_cache, self.attn_tab,
                                      self.n, self.max_rows, self.max_cache, self.out, w.rope_theta,
                                      workspace=self.attn_ws)


# ----------------------------------------------------------------------------- helpers


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed loop runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.15)
        self.proc.terminate()
        self.proc.wait()
        sm, mx, reasons, n = [], [], set(), 0
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                n += 1
                for name, val in zip(("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"),
                                     parts[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": n}


def time_steps(inp: StepInputs, steps: int, warmup: int, dist_on: bool, use_graph: bool = True,
               stages: bool = True):
    """Times K steps.  The step (its five launches) is captured once in a CUDA graph and
    replayed, so the device time is not paced by the host's per-call work.  When a step
    reads less than twice the L2, the L2 is flushed before every timed step, outside that
    step's events.  Returns (total ms of the K steps, per-stage mean ms, description)."""
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        inp.step()
    torch.cuda.synchronize()
    run = inp.step
    if use_graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            inp.step()
        torch.cuda.synchronize()
        for _ in range(warmup):
            graph.replay()
        torch.cuda.synchronize()
        run = graph.replay
    flush = None
    if inp.step_bytes() < 2 * L2_BYTES:
        flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=inp.q.device)
    if dist_on:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    if flush is None:
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for _ in range(steps):
            run()
        t_end.record(stream)
        torch.cuda.synchronize()
        total_ms = t_start.elapsed_time(t_end)
    else:
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for i in range(steps):
            flush.fill_(i & 0x7F)
            evs[i][0].record(stream)
            run()
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        total_ms = sum(a.elapsed_time(b) for a, b in evs)
    if dist_on:
        torch.distributed.barrier()
    stage_ms = time_stages(inp, min(steps, 50), flush) if stages else None
    desc = {"launch": "CUDA graph of the step, replayed" if use_graph else "eager calls",
            "l2": ("inputs larger than L2 (each step reads ~%.0f MB)" % (inp.step_bytes() / 1e6)) if flush is None
            else ("L2 flushed before each timed step (%d MB written outside the step's events; each step reads "
                  "~%.1f MB)" % (FLUSH_BYTES >> 20, inp.step_bytes() / 1e6))}
    return total_ms, stage_ms, desc


def time_stages(inp: StepInputs, reps: int, flush) -> np.ndarray:
    """Per-stage device times of the step as the timed loop runs it: the step is captured once
    more in a CUDA graph with an event-record node between stages (events created `external`),
    and that graph is replayed `reps` times, each replay read back before the next (behind the
    L2 flush where the timed loop flushes).  The kernels then start exactly as in the timed graph,
    with no host time between two events.  Where the installed torch cannot capture timing
    events, each rep runs the step's eager calls behind a GPU-side delay instead, so that the host
    has queued the whole step before the device reaches it (each stage then also holds its
    launch latency).  Mean and median over the reps; the method used is in time_stages.how."""
    ev = None
    graph = None
    try:
        ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(6)]
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            inp.step(ev)
        torch.cuda.synchronize()
        time_stages.how = "CUDA-graph replays of the step with event-record nodes between stages"
    except (TypeError, RuntimeError):
        graph = None
        torch.cuda.synchronize()
        time_stages.how = "eager calls behind a GPU-side delay, events between stages"
    rows = []
    for i in range(reps + 3):
        if flush is not None:
            flush.fill_(i & 0x7F)
        if graph is not None:
            graph.replay()
        else:
            torch.cuda._sleep(SLEEP_CYCLES)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
            inp.step(ev)
        torch.cuda.synchronize()
        if i >= 3:
            rows.append([ev[j].elapsed_time(ev[j + 1]) for j in range(5)])
    a = np.array(rows).reshape(-1, 5)
    time_stages.last_median = np.median(a, axis=0)
    return a.mean(axis=0)


def time_e2e(bufs, steps: int, warmup: int, dist_on: bool):
    """The same step through the public API with host buffers: per step, the step's inputs are
    copied from pinned host memory and the decode result (commit, argmax, conf) is read back.

    With two input sets (`bufs`, each a StepInputs of the same workload) the copies of step
    i + 1 run on a copy stream while step i computes on the current stream (double buffering:
    a buffer is refilled only after the step that read it has finished); with one, copy and
    compute alternate on one stream.  Returns (ms for `steps` steps, bytes in, bytes out per step)."""
    def ins(b):
        return [b.block_tokens, b.topk_ids, b.topk_prob, b.q, b.k, b.v, b.logits]

    def outs(b):
        return [b.commit, b.argmax, b.conf]

    host_in = [t.cpu().pin_memory() for t in ins(bufs[0])]
    host_out = [[torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs(b)] for b in bufs]
    h2d = sum(t.numel() * t.element_size() for t in host_in)
    d2h = sum(t.numel() * t.element_size() for t in host_out[0])
    compute = torch.cuda.current_stream()
    copy = torch.cuda.Stream() if len(bufs) > 1 else compute
    done = [torch.cuda.Event() for _ in bufs]     # the step that read buffer b has finished
    loaded = [torch.cuda.Event() for _ in bufs]   # buffer b holds the next step's inputs
    for e in done:
        e.record(compute)

    def one(i):
        k = i % len(bufs)
        b = bufs[k]
        with torch.cuda.stream(copy):
            copy.wait_event(done[k])
            for d, h in zip(ins(b), host_in):
                d.copy_(h, non_blocking=True)
            loaded[k].record(copy)
        compute.wait_event(loaded[k])
        b.step()
        # the step has read its inputs: the buffer may be refilled (its outputs, read back below,
        # are rewritten only by a later step on this stream); recorded ahead of the read-back,
        # which otherwise queues behind the next copy in and stalls the pipeline
        done[k].record(compute)
        for h, d in zip(host_out[k], outs(b)):
            h.copy_(d, non_blocking=True)

    for i in range(warmup):
        one(i)
    torch.cuda.synchronize()
    if dist_on:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    for i in range(steps):
        one(i)
    torch.cuda.synchronize()
    if dist_on:
        torch.distributed.barrier()
    return (time.perf_counter() - t0) * 1e3, h2d, d2h


# ----------------------------------------------------------------------------- oracle arm


class _RowView:
    """Row access to a bf16 table as float64 without converting the whole table."""

    def __init__(self, t: torch.Tensor):
        self.t = t
        self.shape = tuple(t.shape)

    def __getitem__(self, i):
        return self.t[int(i)].to(torch.float64).numpy()


def oracle_sample(w: W.Workload, budget_s: float, seed: int = 99):
    """Times the CPU oracle on whole denoising steps (selector, sparse input, attention,
    unmasking) of the workload, block indices spread over the sweep, until `budget_s`
    seconds of CPU work are spent.  Returns (steps/s, steps done, seconds, block indices)."""
    from oracle import ssm_oracle as O
    g = torch.Generator().manual_seed(seed)
    V, H = w.vocab, w.hidden
    embed = (torch.randn((V, H), generator=g)).to(torch.bfloat16)
    ev = _RowView(embed)
    mask_id = V - 1
    order = list(w.block_indices)
    if len(order) > 1:
        # spread the sample over the sweep: 0, n/2, n/4, 3n/4, ...
        spread, step = [], len(order)
        seen = set()
        while step >= 1:
            for i in range(0, len(order), step):
                if i not in seen:
                    seen.add(i)
                    spread.append(order[i])
            step //= 2
        order = spread
    done, t_used, used = 0, 0.0, []
    for b in order * max(1, w.batch):
        n_prefix = 0 if w.prefix_cached else w.prompt + b * w.block
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        R = len(r)
        n_new = n_prefix + w.block + R
        n_cache = (w.prompt + b * w.block) if w.prefix_cached else 0
        blk = torch.full((1, w.block), mask_id, dtype=torch.int32)
        ids = torch.randint(0, V - 1, (1, R, w.topk), generator=g)
        probs = torch.softmax(torch.randn((1, R, w.topk), generator=g) * 3, -1).double() * 0.5
        pre = torch.randint(0, V - 1, (1, n_prefix), generator=g) if n_prefix else None
        q = torch.randn((1, n_new, w.h_q, w.head_dim), generator=g).to(torch.bfloat16).double().numpy()
        k = torch.randn((1, n_new, w.h_kv, w.head_dim), generator=g).to(torch.bfloat16).double().numpy()
        v = torch.randn((1, n_new, w.h_kv, w.head_dim), generator=g).to(torch.bfloat16).double().numpy()
        kc = torch.randn((1, n_cache, w.h_kv, w.head_dim), generator=g).to(torch.bfloat16).double().numpy()
        vc = torch.randn((1, n_cache, w.h_kv, w.head_dim), generator=g).to(torch.bfloat16).double().numpy()
        logits = (torch.randn((1, w.block, V), generator=g) * w.logits_sigma).to(torch.bfloat16).double().numpy()
        masked = np.ones((1, w.block), dtype=np.uint8)
        t0 = time.perf_counter()
        r2, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        x, pos = O.build_step_input(ev, mask_id, blk.numpy(), W.block_start(w, b), r2, ids.numpy(), probs.numpy(),
                                    w.alpha, prefix_tokens=None if pre is None else pre.numpy())
        O.attention(q, k, v, pos, kc if n_cache else None, vc if n_cache else None, w.rope_theta)
        O.unmask(logits, masked, O.MODE_THRESHOLD, w.threshold)
        t_used += time.perf_counter() - t0
        done += 1
        used.append(b)
        if t_used >= budget_s:
            break
    return done / t_used, done, t_used, used


def stage_report(inp: "StepInputs", stage_ms, step_ms: float, peaks: dict) -> dict:
    """Per-stage rates and fractions of one measured step, and the step against its floor.

    Fractions: the HBM stages against the measured copy bandwidth by their algorithmic bytes;
    the attention forward and stage against the burst bf16 peak (each is timed on its own, at
    full clock), with the sustained-peak fraction beside it."""
    sel_ms, build_ms, rope_ms, core_ms, unmask_ms = [float(x) for x in stage_ms]
    attn_ms = rope_ms + core_ms
    flops = inp.attn_flops()
    burst = peaks["bf16_tflops"]
    sustained = peaks.get("bf16_tflops_sustained", burst)
    hbm = peaks["hbm_gbs"]
    gb = lambda nbytes, ms: nbytes / (ms * 1e-3) / 1e9 if ms > 0 else 0.0  # noqa: E731
    tf = lambda ms: flops / (ms * 1e-3) / 1e12 if ms > 0 else 0.0  # noqa: E731
    stages = {
        "select_ms": sel_ms, "select": "made inside the gather launch (ssm_select_build_step_input_varlen): "
                                      "select_ms is an empty event pair, build_ms covers both",
        "build_ms": build_ms, "build_GBps": gb(inp.gather_bytes(), build_ms),
        "build_frac_hbm": gb(inp.gather_bytes(), build_ms) / hbm,
        "build_bytes": {"rows_read_distinct": inp.gather_rows_read(), "rows_read_gross": inp.gather_rows_read_gross(),
                        "rows_written": inp.total_rows, "row_bytes": inp.w.hidden * 2,
                        "counted": "distinct embedding rows read once + output rows written"},
        "attention_ms": attn_ms, "attention_TFLOPs": tf(attn_ms),
        "attention_frac_bf16_burst": tf(attn_ms) / burst,
        "attention_frac_bf16_sustained": tf(attn_ms) / sustained,
        "attn_rope_ms": rope_ms, "attn_rope_GBps": gb(inp.rope_bytes(), rope_ms),
        "attn_rope_frac_hbm": gb(inp.rope_bytes(), rope_ms) / hbm,
        "attn_fwd_ms": core_ms, "attn_fwd_TFLOPs": tf(core_ms),
        "attn_fwd_frac_bf16_burst": tf(core_ms) / burst,
        "attn_fwd_frac_bf16_sustained": tf(core_ms) / sustained,
        "attn_fwd_ms_median": float(getattr(time_stages, "last_median", [0.0] * 5)[3]),
        "timing": getattr(time_stages, "how", ""),
        "unmask_ms": unmask_ms, "unmask_GBps": gb(inp.unmask_bytes(), unmask_ms),
        "unmask_frac_hbm": gb(inp.unmask_bytes(), unmask_ms) / hbm,
        "unmask_frac_8TBps_nominal": gb(inp.unmask_bytes(), unmask_ms) / 8000.0,
    }
    # The step's floor: each stage at its own bound (HBM stages at the measured copy bandwidth by
    # their algorithmic bytes, the attention forward at the burst bf16 peak by its algorithmic
    # FLOPs; the selector is launch-latency work and counts as zero), summed over the stages.
    floor_ms = {"build": inp.gather_bytes() / (hbm * 1e9) * 1e3,
                "attn_rope": inp.rope_bytes() / (hbm * 1e9) * 1e3,
                "attn_fwd": flops / (burst * 1e12) * 1e3,
                "unmask": inp.unmask_bytes() / (hbm * 1e9) * 1e3}
    step_floor_ms = sum(floor_ms.values())
    step_roofline = {"ms_per_step": step_floor_ms, "value": inp.n / (step_floor_ms * 1e-3), "unit": UNIT,
                     "frac": step_floor_ms / step_ms, "stage_floor_ms": floor_ms,
                     "how": "sum over stages of algorithmic bytes / measured HBM copy GB/s (build, RoPE pre-pass, "
                            "unmask) and algorithmic FLOPs / measured burst bf16 TFLOP/s (attention forward)"}
    return {"stages": stages, "step_roofline": step_roofline}


def time_eager(inp: "StepInputs", steps: int, warmup: int) -> float:
    """ms per step of eager calls (no CUDA graph), L2 flushed before each step when the
    step's inputs fit in twice the L2 (as the graph replays are timed)."""
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        inp.step()
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=inp.q.device) if inp.step_bytes() < 2 * L2_BYTES \
        else None
    torch.cuda.synchronize()
    total = 0.0
    if flush is None:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            inp.step()
        e1.record(stream)
        torch.cuda.synchronize()
        total = e0.elapsed_time(e1)
    else:
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for i in range(steps):
            flush.fill_(i & 0x7F)
            evs[i][0].record(stream)
            inp.step()
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        total = sum(a.elapsed_time(b) for a, b in evs)
    return total / steps


def measure_configs(dev, steps: int, warmup: int, peaks: dict, skip: str, sweep_steps: int = 10) -> dict:
    """The other workloads, one bench step each as graph replays and as eager calls: denoising
    steps/s, the step-floor fraction, attention TFLOP/s against the burst peak, gather and unmask
    GB/s against the measured copy bandwidth."""
    from paper_2608_23167_gb300 import ssm
    out = {}
    for name in ("tiny", "llada", "dream", "serve", "long"):
        if name == skip:
            continue
        w = W.WORKLOADS[name]
        inp = StepInputs(w, dev)
        torch.cuda.synchronize()
        total_ms, stage_ms, desc = time_steps(inp, steps, warmup, False, use_graph=True)
        eager_ms = time_eager(inp, steps, warmup)
        if ssm.ssm_get_device_error() != 0:
            raise RuntimeError(f"device error in the {name} workload")
        step_ms = total_ms / steps
        rep = stage_report(inp, stage_ms, step_ms, peaks)
        st = rep["stages"]
        out[name] = {
            "workload": workload_desc(w), "denoise_steps_per_bench_step": inp.n, "timed_steps": steps,
            "value": inp.n / (step_ms * 1e-3), "unit": UNIT, "ms_per_step": step_ms,
            "eager_value": inp.n / (eager_ms * 1e-3), "eager_ms_per_step": eager_ms,
            "step_floor_ms": rep["step_roofline"]["ms_per_step"], "step_floor_frac": rep["step_roofline"]["frac"],
            "attention_TFLOPs": st["attention_TFLOPs"], "attention_frac_bf16_burst": st["attention_frac_bf16_burst"],
            "attn_fwd_TFLOPs": st["attn_fwd_TFLOPs"], "attn_fwd_frac_bf16_burst": st["attn_fwd_frac_bf16_burst"],
            "attention_gflop": inp.attn_flops() / 1e9,
            "build_GBps": st["build_GBps"], "build_frac_hbm": st["build_frac_hbm"],
            "unmask_GBps": st["unmask_GBps"], "unmask_frac_hbm": st["unmask_frac_hbm"],
            "stage_ms": {k: st[k] for k in ("select_ms", "build_ms", "attn_rope_ms", "attn_fwd_ms", "unmask_ms")},
            "l2": desc["l2"],
        }
        del inp
        torch.cuda.empty_cache()
        out[name]["sweep"] = time_sweep(w, dev, sweep_steps, warmup)
    return out


def time_sweep(w: W.Workload, dev, steps: int, warmup: int) -> dict:
    """Every block index of the generation, one bench step each (the workload's batch at that
    index), as graph replays behind an L2 flush: the denoising steps of a whole generation
    pass.  Block 0 has the longest suffix; later blocks have shorter suffixes and longer
    prefixes (a longer cache, or without a cache a longer recomputed prefix)."""
    from paper_2608_23167_gb300 import ssm
    per_b = []
    for b in range(w.n_blocks):
        inp = StepInputs(dataclasses.replace(w, block_indices=(b,)), dev)
        total_ms, _, _ = time_steps(inp, steps, warmup, False, use_graph=True, stages=False)
        if ssm.ssm_get_device_error() != 0:
            raise RuntimeError(f"device error in the {w.name} sweep at block {b}")
        per_b.append(total_ms / steps)
        del inp
        torch.cuda.empty_cache()
    tot = sum(per_b)
    return {"blocks": w.n_blocks, "timed_steps_per_block": steps, "ms_per_step_mean": tot / len(per_b),
            "ms_per_step_min": min(per_b), "ms_per_step_max": max(per_b),
            "value": w.batch * len(per_b) / (tot * 1e-3), "unit": UNIT,
            "how": "one graph-replayed step per block index 0..n_blocks-1 (the workload's batch at that index), "
                   "L2 flushed before each; value = denoising steps of the sweep / summed step times"}


def oracle_one_thread(w: W.Workload, budget_s: float) -> dict:
    """The oracle's rate with one host thread: the same sample in a child process whose BLAS
    and OpenMP pools are limited to one thread (they are fixed when numpy loads)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               BLIS_NUM_THREADS="1", NUMEXPR_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    code = ("import json, sys; sys.path.insert(0, %r); import bench; from paper_2608_23167_gb300 import workloads as W; "
            "r = bench.oracle_sample(W.WORKLOADS[%r], %r); print(json.dumps(r[:3]))" % (ROOT, w.name, budget_s))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    if r.returncode != 0:
        return {"value": None, "error": r.stderr.strip().splitlines()[-1:] }
    rate, done, t_used = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{done} whole denoising steps, {t_used:.1f} s of CPU work on one thread"}


def _event_ms(fn, reps: int, warmup: int = 3) -> float:
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def time_next_rows(inp: "StepInputs", attn_ms: float, dev, hbm_peak: float, tensor_peak: float) -> dict:
    """Secondary measurements of the rows that extend the step (not in the timed step).

    unmask_margin / unmask_top1: the unmasking stage of the same step under the margin rule (which
    needs the second-largest probability) and under Vanilla top-1 decoding.
    full_suffix_attention: the attention the same block indices would need without structured
    suffix modeling (every suffix position kept, the dense baseline), and the ratio to the step's
    attention stage.

    suffix_topk: the next step's top-k candidates of every retained suffix position of one bench
    step (this workload's vocabulary, bf16 N(0, sigma) stand-in logits, read once).
    cache_append: the prefix-cache update at block boundaries, 8192 rows of this workload's
    K/V heads (one sequence; 268 MB moved, more than L2) appended into an 8192-row cache.
    """
    from paper_2608_23167_gb300 import ssm
    w = inp.w
    out = {}
    p2 = torch.empty_like(inp.conf)
    for name, kw in (("unmask_margin", dict(p2=p2, mode=ssm.SSM_COMMIT_MARGIN, threshold=w.threshold)),
                     ("unmask_top1", dict(p2=None, mode=ssm.SSM_COMMIT_TOPK, topk=1))):
        ms = _event_ms(lambda: ssm.ssm_unmask(inp.logits, inp.masked, inp.conf, inp.argmax, inp.commit,
                                              workspace=inp.unmask_ws, **kw), reps=20)
        out[name] = {"ms": ms, "GBps": inp.unmask_bytes() / (ms * 1e-3) / 1e9,
                     "frac_hbm": inp.unmask_bytes() / (ms * 1e-3) / 1e9 / hbm_peak}
    if inp.k_cache is not None and w.name == "long":
        # every suffix position of every block index, against the same shared cache
        rows, new_row = [], 0
        for i, b in enumerate(w.block_indices):
            n_new = w.block + (w.n_blocks - 1 - b) * w.block
            rows.append((new_row, inp.cache_row[i], n_new, inp.n_cache[i]))
            new_row += n_new
        fq = W.draw_normal_bf16((new_row, w.h_q, w.head_dim), 1.0, 81, device=dev)
        fk = W.draw_normal_bf16((new_row, w.h_kv, w.head_dim), 1.0, 82, device=dev)
        fv = W.draw_normal_bf16((new_row, w.h_kv, w.head_dim), 1.0, 83, device=dev)
        fpos = torch.cat([torch.arange(W.block_start(w, b), w.prompt + w.gen, dtype=torch.int32)
                          for b in w.block_indices]).to(dev)
        fo = torch.empty_like(fq)
        ftab = ssm.attn_problems_tensor(rows, dev)
        fws = torch.empty(ssm.ssm_attention_workspace_size(new_row, w.h_q, w.h_kv, w.head_dim), dtype=torch.uint8,
                          device=dev)
        max_rows = max(r[2] for r in rows)
        ms = _event_ms(lambda: ssm.ssm_attention_varlen(fq, fk, fv, fpos, inp.k_cache, inp.v_cache, ftab, len(rows),
                                                        max_rows, inp.max_cache, fo, w.rope_theta, workspace=fws),
                       reps=5)
        flops = 4.0 * w.h_q * w.head_dim * sum(r[2] * (r[2] + r[3]) for r in rows)
        out["full_suffix_attention"] = {"rows": new_row, "ms": ms, "gflop": flops / 1e9,
                                        "TFLOPs": flops / (ms * 1e-3) / 1e12,
                                        "frac_bf16": flops / (ms * 1e-3) / 1e12 / tensor_peak,
                                        "ssm_attention_ms": attn_ms, "attention_speedup": ms / attn_ms}
        del fq, fk, fv, fo, fws
    # early termination after a block: one sequence per block index of the sweep, the first block checked
    toks = torch.randint(0, w.vocab - 1, (inp.n, w.gen), dtype=torch.int32, device=dev)
    fin = torch.zeros(inp.n, dtype=torch.uint8, device=dev)
    nact = torch.zeros(1, dtype=torch.int32, device=dev)
    ms = _event_ms(lambda: ssm.ssm_early_stop(toks, w.block, 0, w.vocab - 2, fin, nact), reps=50)
    out["early_stop"] = {"sequences": inp.n, "gen_len": w.gen, "us": ms * 1e3, "bound": "launch latency"}
    del toks, fin, nact
    n = max(inp.total_suffix, 1)
    lg = W.draw_logits((n, w.vocab), inp.w.logits_dtype, w.logits_sigma, 73, device=dev)
    ids = torch.empty((n, w.topk), dtype=torch.int32, device=dev)
    pr = torch.empty((n, w.topk), dtype=torch.float32, device=dev)
    ms = _event_ms(lambda: ssm.ssm_suffix_topk(lg, w.topk, ids, pr), reps=10)
    nbytes = float(n) * w.vocab * lg.element_size()
    out["suffix_topk"] = {"rows": n, "k": w.topk, "ms": ms, "GBps": nbytes / (ms * 1e-3) / 1e9,
                          "frac_hbm": nbytes / (ms * 1e-3) / 1e9 / hbm_peak,
                          "bytes": "the logits of the retained suffix rows, read once"}
    # the step with everything the next step needs from the logits: ssm_unmask_topk (block rows'
    # commits and the retained suffix rows' top-k) in place of ssm_unmask, as graph replays
    logits_pass = lambda: ssm.ssm_unmask_topk(inp.logits, inp.masked, inp.conf, inp.argmax, inp.commit, lg,  # noqa: E731
                                              w.topk, ids, pr, threshold=w.threshold, min_commit=1,
                                              workspace=inp.unmask_ws)
    ms_lp = _event_ms(logits_pass, reps=10)
    lp_bytes = inp.unmask_bytes() + nbytes
    eager_ms = _event_ms(lambda: inp.step(unmask=logits_pass), reps=20)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        inp.step(unmask=logits_pass)
    torch.cuda.synchronize()
    step_ms = _event_ms(graph.replay, reps=20)
    del graph
    out["step_with_suffix_topk"] = {
        "value": inp.n / (step_ms * 1e-3), "unit": UNIT, "ms_per_step": step_ms,
        "eager_value": inp.n / (eager_ms * 1e-3), "eager_ms_per_step": eager_ms,
        "logits_ms": ms_lp, "logits_GBps": lp_bytes / (ms_lp * 1e-3) / 1e9,
        "logits_frac_hbm": lp_bytes / (ms_lp * 1e-3) / 1e9 / hbm_peak,
        "how": "the step with ssm_unmask_topk over the block rows' and the retained suffix rows' logits in place "
               "of ssm_unmask, captured once in a CUDA graph and replayed back to back (eager_*: the same step as "
               "direct calls); logits_* is that call alone (its bytes: both sets of logits, read once)"}
    del lg, ids, pr
    n = 8192
    kn = W.draw_normal_bf16((1, n, w.h_kv, w.head_dim), 1.0, 71).to(dev)
    vn = W.draw_normal_bf16((1, n, w.h_kv, w.head_dim), 1.0, 72).to(dev)
    kc = torch.empty_like(kn)
    vc = torch.empty_like(vn)
    pos = torch.arange(n, dtype=torch.int32, device=dev)
    ms = _event_ms(lambda: ssm.ssm_cache_append(kn, vn, pos, kc, vc, 0, w.rope_theta), reps=20)
    nbytes = 4.0 * n * w.h_kv * w.head_dim * 2
    out["cache_append"] = {"rows": n, "ms": ms, "GBps": nbytes / (ms * 1e-3) / 1e9,
                           "frac_hbm": nbytes / (ms * 1e-3) / 1e9 / hbm_peak,
                           "bytes": "K and V rows read once and written once (rotated K)"}
    del kn, vn, kc, vc
    return out


def reduce_max(x: float, device, dist_on: bool) -> float:
    """Max over ranks of a per-rank time (the job ends when its slowest replica ends)."""
    if not dist_on:
        return float(x)
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def run_reference(args, w: W.Workload, rank: int):
    if rank != 0:
        return
    budget = max(1.0, float(os.environ.get("SSM_ORACLE_STEP_BUDGET_S", "8")))
    rates = []
    for _ in range(args.warmup):
        oracle_sample(w, min(budget, 2.0))
    t_total = 0.0
    done_total = 0
    for _ in range(args.steps):
        rate, done, t, used = oracle_sample(w, budget)
        rates.append(rate)
        t_total += t
        done_total += done
    value = done_total / t_total
    sample = (f"per bench step: whole denoising steps of the '{w.name}' workload on block indices spread over "
              f"the sweep until {budget:.0f} s of CPU work; {done_total} denoising steps in {t_total:.1f} s")
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * t_total / max(args.steps, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": workload_desc(w), "parallelism": "replicas"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": host_cores(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def workload_desc(w: W.Workload) -> str:
    blocks = (f"block indices {w.block_indices[0]}..{w.block_indices[-1]} as one batch"
              if len(w.block_indices) > 1 else f"block index {w.block_indices[0]}")
    cache = "prompt in a prefix KV cache" if w.prefix_cached else "prompt recomputed (no cache)"
    return (f"{w.name}: {w.h_q}/{w.h_kv} heads, head_dim {w.head_dim}, hidden {w.hidden}, prompt {w.prompt} "
            f"({cache}), gen {w.gen}, block {w.block}, budgets local {w.local}/middle {w.middle}/tail {w.tail}, "
            f"batch {w.batch}, {blocks}, vocab {w.vocab} {w.logits_dtype} logits, top-k {w.topk}, alpha {w.alpha}, "
            f"threshold {w.threshold}")


# ----------------------------------------------------------------------------- main


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ssm", "reference"], default="ssm")
    ap.add_argument("--workload", default="long", choices=list(W.WORKLOADS))
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="time eager calls instead of a captured CUDA graph")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-next", action="store_true", help="skip the secondary measurements of the next rows")
    ap.add_argument("--no-configs", action="store_true", help="skip the per-workload block of the other workloads")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    w = W.WORKLOADS[args.workload]
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, w, rank)
        return

    dist_on = world > 1
    torch.cuda.set_device(local_rank)
    if dist_on:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    from paper_2608_23167_gb300 import build_lib, ssm
    if rank == 0 or not dist_on:
        build_lib.build()
    if dist_on:
        torch.distributed.barrier()
    ssm.lib()
    dev = torch.device("cuda", local_rank)
    inp = StepInputs(w, dev)
    torch.cuda.synchronize()

    clocks = ClockSampler(local_rank)
    clocks.start()
    total_ms, stage_ms, timing_desc = time_steps(inp, args.steps, args.warmup, dist_on, use_graph=not args.no_graph)
    clk = clocks.stop()
    err = ssm.ssm_get_device_error()
    if err != 0:
        raise RuntimeError(f"device error {err} during the timed region")

    total_ms = reduce_max(total_ms, dev, dist_on)
    n_per_step = inp.n
    units = inp.n * args.steps * world                 # denoising steps processed by all ranks
    value = units / (total_ms / 1e3)

    e2e = None
    if not args.no_e2e:
        # a second input set for double buffering (the embedding table, cache and workspaces are
        # per set too: about 3 GB for the long sweep)
        inp2 = StepInputs(w, dev)
        e_ms, h2d, d2h = time_e2e([inp, inp2], args.steps, min(args.warmup, 5), dist_on)
        del inp2
        torch.cuda.empty_cache()
        e_ms = reduce_max(e_ms, dev, dist_on)
        e2e = {"value": inp.n * args.steps * world / (e_ms / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "how": "host clock over the steps; per step its inputs copied from pinned host memory (on a copy "
                      "stream, into one of two input sets, while the previous step computes) and commit, argmax "
                      "and conf read back"}

    peaks, peak_src = load_peaks()
    rep = stage_report(inp, stage_ms, total_ms / args.steps, peaks)
    flops = inp.attn_flops()
    traffic = None
    tpath = os.path.join(ROOT, "profiles", f"attention_{w.name}_traffic.json")
    if os.path.exists(tpath):
        with open(tpath) as f:
            tr = json.load(f)
        part = tr.get("parts", {}).get("attn_fwd_kernel")
        if tr.get("source_digest") == build_lib.source_digest(*build_lib.ATTENTION_SOURCES) and part:
            traffic = (part["dram_read_MB"] + part["dram_write_MB"]) * 1e6
    # the forward timed alone: back-to-back launches of the step's forward (its inputs as the
    # step leaves them) between two events on its stream, so that the events' own gaps do not
    # count; the kernel runs at full clock, so its fraction is taken against the burst bf16 peak
    # (the sustained figure, a power-capped GEMM loop, is reported beside it).  The forward's
    # time inside the step (an event-record node on each side) is in stages.attn_fwd_ms.
    from paper_2608_23167_gb300 import ssm as _ssm
    fwd_reps = 20
    fwd_ms = _event_ms(inp.attn_core, reps=fwd_reps)
    if _ssm.ssm_get_device_error() != 0:
        raise RuntimeError("device error while timing the forward alone")
    core_tflops = flops / (fwd_ms * 1e-3) / 1e12
    roofline = {"bound": "tensor", "achieved": core_tflops, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": core_tflops / peaks["bf16_tflops"], "traffic": traffic,
                "kernel": "attn_fwd_kernel (ssm_attention_varlen_core)",
                "peak_kind": f"bf16 dense, burst ({peak_src})",
                "frac_of_sustained_peak": core_tflops / peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"]),
                "launch_ms": fwd_ms,
                "timing": f"{fwd_reps} back-to-back launches between two CUDA events on the launching stream",
                "in_step": {"ms": rep["stages"]["attn_fwd_ms"], "frac": rep["stages"]["attn_fwd_frac_bf16_burst"],
                            "how": "inside the step, an event-record node on each side"},
                "algorithmic": f"{flops / 1e9:.1f} GFLOP per launch = 4 * heads * head_dim * sum(Nq * Nk)"}
    stages = rep["stages"]
    step_roofline = rep["step_roofline"]
    hbm_peak = peaks["hbm_gbs"]
    tensor_peak = peaks["bf16_tflops"]
    attn_ms = stages["attention_ms"]

    # the same step as eager calls (no CUDA graph): what a caller without graph capture gets
    eager_ms = time_eager(inp, min(args.steps, 100), args.warmup)
    eager = {"value": inp.n / (eager_ms * 1e-3), "unit": UNIT, "ms_per_step": eager_ms,
             "steps": min(args.steps, 100)}

    next_rows = None
    if rank == 0 and not args.no_next:
        next_rows = time_next_rows(inp, attn_ms, dev, hbm_peak, tensor_peak)
        if ssm.ssm_get_device_error() != 0:
            raise RuntimeError("device error in the secondary measurements")

    configs = None
    if rank == 0 and world == 1 and not args.no_configs:
        del inp
        torch.cuda.empty_cache()
        configs = measure_configs(dev, min(args.steps, 100), args.warmup, peaks, skip=w.name)
        inp = None

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        budget = float(os.environ.get("SSM_CPU_BASELINE_BUDGET_S", "15"))
        rate, done, t_used, used = oracle_sample(w, budget)
        cpu = {"value": rate, "unit": UNIT, "cores": host_cores(), "kind": "oracle",
               "sample": f"{done} whole denoising steps (block indices {used}) of the same workload, "
                         f"{t_used:.1f} s of CPU work, numpy fp64 with its default BLAS threads",
               "one_thread": oracle_one_thread(w, float(os.environ.get("SSM_CPU_1T_BUDGET_S", "8")))}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": workload_desc(w), "denoise_steps_per_bench_step": n_per_step,
                       "parallelism": "replicas" if world > 1 else "single GPU", **timing_desc},
            "roofline": roofline, "step_roofline": step_roofline, "stages": stages, "clocks": clk, "e2e": e2e,
            "cpu_baseline": cpu, "gpu_launches": StepInputs.LAUNCHES_PER_STEP * args.steps,
            "eager": eager, "next_rows": next_rows, "configs": configs,
        }
        print(json.dumps(line), flush=True)
    if dist_on:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
