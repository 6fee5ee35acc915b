#!/usr/bin/env python3
"""Benchmark: SDSAT two-step-draft-then-verify decoding on GB300 (one JSON line).

A step is one block decode step: build the block input, one block forward of
q = k + 1 positions through every layer, target selection + Eq. 3 verification
+ KV commit.  Steps alternate draft step 1 / draft step 2 (Sec. 2.1.1); a
generation is the steps that emit `new` tokens per sequence after a `prompt`
of uniform ids, and generations run back to back.  Drafts come from a seeded
per-position stub that copies the model's own plain-decoding token with the
workload's match rate (random weights cannot draft).

value      generated tokens/s, the loop replayed from CUDA graphs, inputs and
           state resident in HBM (weights 13-26 GB > L2, so no flush needed).
e2e        the same metric through the C ABI with host buffers: each step the
           host builds the block input, copies it in (pinned -> device), runs the
           step, copies the emitted tokens back and reads them.
roofline   the skinny GEMM (the dominant kernel): algorithmic bytes / CUDA-event
           time of its launches in a profiled pass, against the measured HBM
           copy bandwidth.
cpu_baseline / --impl reference   the CPU oracle timed on a bounded sample.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "generated tokens/s at bs1 (7B/13B shape); verify-step HBM GB/s vs 8 TB/s"
NOMINAL_HBM_GBS = 8000.0

WORKLOADS = {
    # CodeLlama-7B shape, greedy, prompt 2048, 256 new tokens, k = 5, stub match 0.7
    "7b": dict(shape="7b", batch=1, prompt=2048, new=256, k=5, temperature=0.0, top_p=1.0, top_k=0, match=0.7),
    # CodeLlama-13B shape, greedy, prompt 4096
    "13b": dict(shape="13b", batch=1, prompt=4096, new=256, k=5, temperature=0.0, top_p=1.0, top_k=0, match=0.7),
    # 7B shape, nucleus verification (top_p 0.95, T 0.2), batch 4, prompts of 1024
    "7b-nucleus": dict(shape="7b", batch=4, prompt=1024, new=256, k=5, temperature=0.2, top_p=0.95, top_k=0,
                       match=0.6),
    # 7B shape, tree draft step 2 (Sec. 2.1.2): nucleus T 0.2, top_p 0.95, top_k 10 (the paper's
    # nucleus setting), k = 5 = tree depth, two chains of drafts below the root (q = 11)
    "7b-tree": dict(shape="7b", batch=1, prompt=2048, new=256, k=5, temperature=0.2, top_p=0.95, top_k=10,
                    match=0.6, width=2, match2=0.4),
    # 7B shape, greedy, the pipelined variant (not a step of the paper): every block carries
    # y, the k drafts and the k adaptive tokens (q = 2k + 1); a fully accepted block skips
    # the next draft step 1
    "7b-pipelined": dict(shape="7b", batch=1, prompt=2048, new=256, k=5, temperature=0.0, top_p=1.0, top_k=0,
                         match=0.7, pipelined=True),
    # tiny correctness shape
    "tiny": dict(shape="tiny", batch=1, prompt=128, new=64, k=5, temperature=0.0, top_p=1.0, top_k=0, match=0.7),
}


# DRAM bytes (read + write) per algorithmic byte of the skinny GEMM, from one ncu capture
# (--set full) of a gate/up-sized launch: K 4096, N 22016, M 6 -> 186.01 MB of traffic for
# 180.98 MB of weights + operand + output.  The bench line applies it to the step's gate/up
# launch (the roofline's kernel).  GEMM_TRAFFIC_CURRENT says whether that capture was taken of
# the kernel as it is now; while it is False the line reports traffic null.
GEMM_TRAFFIC_RATIO = 186.01 / 180.98
GEMM_TRAFFIC_CURRENT = True
GEMM_TRAFFIC_SOURCE = ("ncu dram__bytes_read+write of one K=4096 N=22016 M=6 launch (186.01 MB for 180.98 MB "
                       "algorithmic, profiles/gemm_gateup_4096x22016_m6.md) times the gate/up launch's algorithmic "
                       "bytes; bytes per launch")


def expected_tokens_per_step(k: int, match: float, matches=None) -> float:
    """Two steps emit 2 + m tokens, m = leading matches of k drafts (Sec. 2.1.1); with several
    branches of independent stub coins (match rates `matches`), m is the longest accepted branch:
    P(m >= i) = 1 - prod_w (1 - p_w^i)."""
    ps = list(matches) if matches else [match]
    tail = 0.0
    for i in range(1, k + 1):
        miss = 1.0
        for p in ps:
            miss *= 1.0 - p ** i
        tail += 1.0 - miss
    return (2.0 + tail) / 2.0


def expected_tokens_per_step_pipelined(k: int, match: float) -> float:
    """Pipelined blocks (stub coins with rate `match`): a mode-A block emits 1 + m and stays
    in mode A iff m = k (probability p^k), a mode-S block emits 1 and leads to mode A;
    stationary mean tokens per block."""
    pk = match ** k
    pi_a = 1.0 / (2.0 - pk)
    return pi_a * (1.0 + sum(match ** i for i in range(1, k + 1))) + (1.0 - pi_a)


def branch_matches(wl):
    """Stub match rate of every branch of the workload's draft tree (one branch: the chain)."""
    w = wl.get("width", 1)
    return [wl["match"]] + [wl.get("match2", wl["match"])] * (w - 1)


def chains_parent(width: int, k: int):
    """Parent rows of the draft tree of `width` chains of k drafts below the root (row 0)."""
    return [-1] + [0 if i == 0 else 1 + w * k + i - 1 for w in range(width) for i in range(k)]


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def tensor_peak():
    """Dense bf16 tensor-core peak (TFLOP/s): the measured burst cuBLAS figure, else the fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.proc = None
        self.uuid = uuid

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits", "-lms", "100"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            return None
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- bytes
def gemm_bytes(shape, M):
    """Algorithmic HBM bytes of one launch of each projection (weights + activations + outputs)."""
    d, F, R, V = shape.d_model, shape.ffn_dim, shape.n_heads * shape.head_dim, shape.vocab
    return {
        "gemm_qkv": 3 * R * d * 2 + M * d * 4 + M * R * 4 + 2 * M * R * 2,
        "gemm_o": d * R * 2 + M * R * 4 + 2 * M * d * 4,
        "gemm_gateup": 2 * F * d * 2 + M * d * 4 + M * F * 4,
        "gemm_down": d * F * 2 + M * F * 4 + 2 * M * d * 4,
        "gemm_lm_head": V * d * 2 + M * d * 4 + M * V * 4,
    }


def weight_bytes(shape):
    d, F, R, V, L = shape.d_model, shape.ffn_dim, shape.n_heads * shape.head_dim, shape.vocab, shape.n_layers
    return L * (4 * R * d + 3 * F * d) * 2 + 2 * V * d * 2


def kv_bytes_per_layer_slot(shape):
    return 2 * shape.n_heads * shape.head_dim * 2


# ----------------------------------------------------------------------------- our arm
def shard_sequences(rank, b):
    """The sequence ids rank `rank` decodes: each rank of a replica run takes its own b
    sequences (own prompts and draft stubs), so ranks share no data and need no collective."""
    return [rank * b + s for s in range(b)]


def combine_ranks(ms, tokens, world, device):
    """Whole-job (time, tokens) of a replica run: the slowest rank's time and every rank's
    tokens (value = tokens / time)."""
    if world == 1:
        return ms, tokens
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms), float(tokens)], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return mx[0].item(), t[1].item()


class Runner:
    def __init__(self, wl, device, weights=None, shard=0):
        import torch
        import synth
        import paper_2403_18647_gb300 as sd
        self.torch, self.synth, self.sd = torch, synth, sd
        self.wl = wl
        self.shape = synth.SHAPES[wl["shape"]]
        self.b, self.k = wl["batch"], wl["k"]
        self.pipe = bool(wl.get("pipelined"))
        self.kinds = 1 if self.pipe else 2        # step kinds of a loop (graphs)
        self.q = 2 * self.k + 1 if self.pipe else self.k + 1   # draft step 1 block rows (pipelined: every block)
        self.width = wl.get("width", 1)
        self.tree = self.width > 1
        self.q2 = self.q if self.pipe else 1 + self.width * self.k   # draft step 2 block rows (chain: q)
        self.qmax = max(self.q, self.q2)
        self.P = wl["prompt"]
        self.new = wl["new"]
        self.cap = self.P + 2 * self.new + 8 * self.qmax
        self.dev = device
        self.weights = weights if weights is not None else synth.make_model(self.shape, seed=wl.get("seed", 0),
                                                                            device=device)
        torch.cuda.synchronize()
        self.ctx = sd.Context(self.shape, self.weights, max_position=self.cap + 64)
        self.kv = self.ctx.kv(self.b, self.cap)
        V = self.shape.vocab
        self.logits = torch.empty(self.b * self.qmax, V, device=device)
        self.toks = torch.zeros(self.b * self.qmax, dtype=torch.int32, device=device)
        self.acc = torch.ones(self.b, dtype=torch.int32, device=device)
        self.out = torch.zeros(self.b * self.qmax, dtype=torch.int32, device=device)
        self.parent = torch.tensor(chains_parent(self.width, self.k) * self.b, dtype=torch.int32, device=device)
        self.pmode = torch.ones(self.b, dtype=torch.int32, device=device)    # pipelined: the previous block's mode
        self.pnver = torch.zeros(self.b, dtype=torch.int32, device=device)
        self.seq_ids = shard_sequences(shard, self.b)
        self.prompts = [synth.prompt_ids(0, i, self.P, self.shape.adaptive_id, device) for i in self.seq_ids]
        for s in range(self.b):
            self.ctx.prefill(self.kv, s, self.prompts[s][:-1].contiguous())
        self.prefill_ms = self._time_prefill()
        self.first = torch.stack([p[-1] for p in self.prompts]).to(torch.int32)
        # the loop starts as if a draft step 2 block (q2 rows) had just emitted the last prompt token
        self.init_out = torch.zeros_like(self.out)
        for s in range(self.b):
            self.init_out[s * self.q2] = self.prompts[s][-1]
        self.init_acc = torch.ones_like(self.acc)
        self.start_len = torch.full((self.b,), self.P - 1, dtype=torch.int32, device=device)
        self._make_table()
        torch.cuda.synchronize()

    def _time_prefill(self, reps=3):
        """Device time of sequence 0's prompt prefill (the step before the decode loop), rerun
        from an empty cache after the first, untimed one."""
        torch = self.torch
        lens = self.ctx.kv_lengths(self.kv).clone()
        zero = lens.clone()
        zero[0] = 0
        toks = self.prompts[0][:-1].contiguous()
        times = []
        for _ in range(reps):
            self.ctx.kv_commit(self.kv, zero, self.b)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            self.ctx.prefill(self.kv, 0, toks)
            e1.record()
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1))
        self.ctx.kv_commit(self.kv, lens, self.b)
        return min(times)

    # target selection for this workload
    def accept(self, n_verify, commit=True):
        wl = self.wl
        if wl["temperature"] > 0:
            self.ctx.accept_nucleus(self.kv, self.logits, self.toks, self.b, self.q, n_verify, wl["top_p"],
                                    wl["temperature"], 1234, self.acc, self.out, top_k=wl["top_k"], commit=commit)
        else:
            self.ctx.accept_greedy(self.kv, self.logits, self.toks, self.b, self.q, n_verify, self.acc, self.out,
                                   commit=commit)

    def _make_table(self):
        """Plain decoding (q = 1) from the prompt gives each position's reference token; the stub
        table holds it with the workload's match rate, else a uniform id."""
        torch = self.torch
        n_ref = 2 * self.new + 8 * self.q
        ref = torch.zeros(n_ref, self.b, dtype=torch.int32, device=self.dev)
        lg = torch.empty(self.b, self.shape.vocab, device=self.dev)
        tok = self.first.clone()
        acc = torch.empty(self.b, dtype=torch.int32, device=self.dev)
        wl = self.wl
        n_run = min(n_ref, self.cap - self.P)
        for i in range(n_run):
            self.ctx.block_forward(self.kv, tok, lg, self.b, 1)
            if wl["temperature"] > 0:
                self.ctx.accept_nucleus(self.kv, lg, tok, self.b, 1, 0, wl["top_p"], wl["temperature"], 1234, acc,
                                        tok, top_k=wl["top_k"])
            else:
                self.ctx.accept_greedy(self.kv, lg, tok, self.b, 1, 0, acc, tok)
            ref[i] = tok
        self.ctx.kv_commit(self.kv, self.start_len, self.b)
        self.stride = self.cap + 32
        # [width][b][stride]: branch w's stub (own coins) with its match rate
        table = torch.zeros(self.width, self.b, self.stride, dtype=torch.int32, device=self.dev)
        for w, match in enumerate(branch_matches(wl)):
            for s in range(self.b):
                full = torch.zeros(self.stride, dtype=torch.int32, device=self.dev)
                full[self.P:self.P + n_run] = ref[:n_run, s]
                table[w, s] = self.synth.stub_table(w, self.seq_ids[s], full, match, self.shape.vocab)
        self.table = table.contiguous()
        self.ref = ref

    def reset(self):
        self.ctx.kv_commit(self.kv, self.start_len, self.b)
        self.out.copy_(self.init_out)
        self.acc.copy_(self.init_acc)
        self.pmode.fill_(1)

    def step(self, mode):
        if self.pipe:
            wl = self.wl
            self.ctx.build_pipelined_block(self.kv, self.out, self.acc, self.pmode, self.pnver, self.toks, self.b,
                                           self.k, draft_table=self.table, table_stride=self.stride)
            self.ctx.block_forward(self.kv, self.toks, self.logits, self.b, self.q)
            self.ctx.accept_pipelined(self.kv, self.logits, self.toks, self.pnver, self.b, self.q, self.acc, self.out,
                                      temperature=wl["temperature"], top_p=wl["top_p"], seed=1234, top_k=wl["top_k"])
            return
        if not self.tree:
            self.ctx.build_block(self.kv, mode, self.out, self.acc, self.toks, self.b, self.q,
                                 draft_table=self.table if mode == 2 else None, table_stride=self.stride)
            self.ctx.block_forward(self.kv, self.toks, self.logits, self.b, self.q)
            self.accept(0 if mode == 1 else self.k)
        elif mode == 1:
            self.ctx.build_tree_block(self.kv, 1, self.out, self.q2, self.acc, self.toks, self.b, self.k)
            self.ctx.block_forward(self.kv, self.toks, self.logits, self.b, self.q)
            self.accept(0)
        else:
            self.ctx.build_tree_block(self.kv, 2, self.out, self.q, self.acc, self.toks, self.b, self.k,
                                      draft_tables=self.table, width=self.width, table_stride=self.stride)
            self.forward_accept_tree()

    def forward_accept_tree(self):
        """Draft step 2 as a tree (Sec. 2.1.2): tree forward, then tree verification, compaction
        of the accepted branch's KV rows and commit."""
        wl = self.wl
        self.ctx.block_forward_tree(self.kv, self.toks, self.parent, self.logits, self.b, self.q2)
        self.ctx.accept_tree(self.kv, self.logits, self.toks, self.parent, self.b, self.q2, self.acc, self.out,
                             temperature=wl["temperature"], top_p=wl["top_p"], seed=1234, top_k=wl["top_k"])

    def calibrate(self):
        """One generation with host checks: the number of steps it takes and the tokens
        and committed lengths of every step (for the byte counts)."""
        torch = self.torch
        self.reset()
        base = self.ctx.kv_emitted(self.kv).clone()
        lens, toks = [], []
        n = 0
        while True:
            lens.append(self.ctx.kv_lengths(self.kv).cpu().tolist())
            self.step(1 if n % 2 == 0 else 2)
            n += 1
            em = (self.ctx.kv_emitted(self.kv) - base).cpu().tolist()
            toks.append(sum(em) - sum(toks))
            if n % self.kinds == 0 and min(em) >= self.new:
                break
        flags = self.ctx.get_error()
        return n, lens, toks, flags

    def capture(self):
        torch = self.torch
        try:
            graphs = []
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(s):
                for mode in (1, 2)[:self.kinds]:   # warm the path on the capture stream
                    self.step(mode)
            torch.cuda.current_stream().wait_stream(s)
            torch.cuda.synchronize()
            for mode in (1, 2)[:self.kinds]:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    self.step(mode)
                graphs.append(g)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                self.reset()
            graphs.append(g)
            torch.cuda.synchronize()
            return graphs
        except Exception as e:  # graphs are an optimisation; eager launches run the same kernels
            print("note: CUDA graph capture failed (%s); timing eager launches" % e, file=sys.stderr)
            torch.cuda.synchronize()
            return None

    def run_steps(self, n, steps_per_gen, graphs, start=0):
        """n steps of back-to-back generations, starting at global step index `start`."""
        for i in range(start, start + n):
            j = i % steps_per_gen
            if j == 0 and i > 0:
                graphs[self.kinds].replay() if graphs else self.reset()
            if graphs:
                graphs[j % self.kinds].replay()
            else:
                self.step(1 if j % 2 == 0 else 2)


def accept_rate(r, toks):
    """Mean fraction of the k drafts accepted per verify step (draft step 2), from one
    calibrated generation: a verify step emits 1 + m tokens per sequence."""
    if r.pipe:   # every block: the mean fraction of k accepted over the blocks that verified
        return None
    ver = [t for i, t in enumerate(toks) if i % 2 == 1]
    if not ver:
        return None
    return round(statistics.mean((t / r.b - 1.0) / r.k for t in ver), 4)


def step_latency(r, graphs, steps_per_gen, n):
    """Per block step device latency (CUDA events around each replay): p10 / median / p90 in ms."""
    torch = r.torch
    if not graphs:
        return None
    r.reset()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    torch.cuda.synchronize()
    ev[0].record()
    for i in range(n):
        j = i % steps_per_gen
        if j == 0 and i > 0:
            graphs[r.kinds].replay()
        graphs[j % r.kinds].replay()
        ev[i + 1].record()
    torch.cuda.synchronize()
    t = sorted(ev[i].elapsed_time(ev[i + 1]) for i in range(n))
    pick = lambda f: round(t[min(n - 1, int(f * n))], 4)
    return {"p10": pick(0.1), "median": pick(0.5), "p90": pick(0.9), "steps": n}


def run_plain(r, steps, warmup=3):
    """The in-build baseline: plain decoding (q = 1, one token per forward) through the same
    kernels, CUDA-graph replayed; tokens/s over `steps` forwards from the prompt."""
    torch = r.torch
    b, V, wl = r.b, r.shape.vocab, r.wl
    steps = min(steps, r.new)
    tok = torch.empty(b, dtype=torch.int32, device=r.dev)
    lg = torch.empty(b, V, device=r.dev)
    acc = torch.empty(b, dtype=torch.int32, device=r.dev)

    def init():
        r.ctx.kv_commit(r.kv, r.start_len, b)
        tok.copy_(r.first)

    def step():
        r.ctx.block_forward(r.kv, tok, lg, b, 1)
        if wl["temperature"] > 0:
            r.ctx.accept_nucleus(r.kv, lg, tok, b, 1, 0, wl["top_p"], wl["temperature"], 1234, acc, tok,
                                 top_k=wl["top_k"])
        else:
            r.ctx.accept_greedy(r.kv, lg, tok, b, 1, 0, acc, tok)

    init()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for _ in range(warmup):
            step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    init()
    for _ in range(warmup):
        g.replay()
    init()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    init()
    return {"tokens_per_s": round(b * steps / (ms / 1e3), 2), "ms_per_step": round(ms / steps, 4), "steps": steps,
            "note": "plain greedy/nucleus decoding, q = 1, same kernels and graphs (in-build baseline)"}


def run_ours(args, wl, rank, world):
    import torch
    import torch.distributed as dist
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    r = Runner(wl, dev, shard=rank)
    shape = r.shape
    steps_per_gen, lens, toks_cal, flags = r.calibrate()
    # schedule the timed region as whole-generation-aligned steps
    graphs = r.capture()
    r.reset()
    r.run_steps(args.warmup, steps_per_gen, graphs)
    r.reset()
    torch.cuda.synchronize()
    em0 = r.ctx.kv_emitted(r.kv).sum().item()
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        pass
    clocks = ClockSampler(uuid)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push("bench:timed")   # lets a profiler restrict itself to the timed steps
    e0.record()
    r.run_steps(args.steps, steps_per_gen, graphs)
    e1.record()
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1)
    tokens = r.ctx.kv_emitted(r.kv).sum().item() - em0
    flags |= r.ctx.get_error()
    ms, tokens = combine_ranks(ms, tokens, world, dev)
    value = tokens / (ms / 1e3)
    # --- profiled pass (per-kernel CUDA events; launches serialised) for the roofline
    r.reset()
    n_prof = min(args.steps, steps_per_gen)
    launches_per_step = 4 + 5 * shape.n_layers   # build, embed+norm, 5 per layer, head, accept
    r.ctx.profile_begin(n_prof * (launches_per_step + 2) + 16)
    r.run_steps(n_prof, steps_per_gen, None)
    kstats = r.ctx.profile_end()
    # --- per-step latency percentiles and the plain-decoding baseline on the same kernels
    lat = step_latency(r, graphs, steps_per_gen, min(args.steps, 4 * steps_per_gen))
    plain = run_plain(r, min(args.steps, 128))
    # --- e2e: the C ABI with host buffers (host builds inputs, reads outputs every step)
    e2e = run_e2e(r, args.steps, steps_per_gen)
    # --- bytes (steps alternate q-row and q2-row blocks; for the chain q2 = q)
    rows = [r.q if i % 2 == 0 else r.q2 for i in range(len(lens))]
    gb1, gb2 = gemm_bytes(shape, r.b * r.q), gemm_bytes(shape, r.b * r.q2)
    gb = {n: (gb1[n] + gb2[n]) / 2.0 for n in gb1}
    g_bytes = sum(gb[n] * kstats.get(n, (0, 0))[0] for n in gb)
    g_ms = sum(kstats.get(n, (0, 0.0))[1] for n in gb)
    g_launches = sum(kstats.get(n, (0, 0))[0] for n in gb)
    peak, peak_kind = peaks()
    achieved = g_bytes / (g_ms / 1e3) / 1e9 if g_ms > 0 else 0.0
    # the launch with the largest share of the step's device time: gate/up
    gu_n, gu_ms = kstats.get("gemm_gateup", (0, 0.0))
    gu_bytes = gb["gemm_gateup"]
    gu_achieved = gu_bytes / (gu_ms / gu_n / 1e3) / 1e9 if gu_n and gu_ms > 0 else 0.0
    prof_ms = sum(v[1] for v in kstats.values())
    # per-step algorithmic bytes over one calibrated generation
    Wb = weight_bytes(shape)
    slot = kv_bytes_per_layer_slot(shape) * shape.n_layers
    kv_read = [sum(l + q for l in ln) * slot for ln, q in zip(lens, rows)]
    kv_write = [r.b * q * slot for q in rows]
    logit_b = [r.b * q * shape.vocab * 4 for q in rows]
    step_bytes = Wb + statistics.mean(kv_read) + statistics.mean(kv_write) + statistics.mean(logit_b)
    ms_step = ms / args.steps
    step_gbs = step_bytes / (ms_step / 1e3) / 1e9
    # --- gpu launches in the timed region: our kernels only (a tree step adds its prep and
    # compaction kernels)
    resets = sum(1 for i in range(args.steps) if i % steps_per_gen == 0 and i > 0)
    tree_steps = sum(1 for i in range(args.steps) if (i % steps_per_gen) % 2 == 1) if r.tree else 0
    gpu_launches = args.steps * launches_per_step + 2 * tree_steps + resets
    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": args.config, "model": shape.name + "-shaped random init (seed %d)" % wl.get("seed", 0),
                   "global_batch": r.b * world, "seq_len": r.P, "new_tokens": r.new, "k": r.k, "q": r.q,
                   "draft_stub_match": branch_matches(wl) if r.tree else wl["match"],
                   "temperature": wl["temperature"], "top_p": wl["top_p"], "top_k": wl["top_k"],
                   "parallelism": "replicas%d" % world if world > 1 else "single",
                   "l2": "inputs larger than L2 (%.1f GB of weights streamed per step)" % (Wb / 1e9),
                   "graphs": graphs is not None, "mma": "bf16 hi+lo activations x bf16 weights -> fp32"},
        "tokens_per_step": round(tokens / world / args.steps, 4),
        "tokens_per_step_basis": "tokens emitted in the timed window (a fixed run of steps from the start of "
                                 "back-to-back generations, so it varies with the window's length)",
        "tokens_per_step_generation": round(sum(toks_cal) / len(toks_cal), 4),
        "value_generation_basis": round(world * sum(toks_cal) / len(toks_cal) / (ms / args.steps / 1e3), 2),
        "value_expected_basis": round(world * r.b * (expected_tokens_per_step_pipelined(r.k, wl["match"]) if r.pipe
                                                      else expected_tokens_per_step(r.k, wl["match"],
                                                                                    branch_matches(wl)))
                                      / (ms / args.steps / 1e3), 2),
        "accept_rate": accept_rate(r, toks_cal),
        "step_latency_ms": lat,
        "plain_decoding": plain,
        "speedup_vs_plain": round(value / world / plain["tokens_per_s"], 3) if plain else None,
        "expected_tokens_per_step": round(expected_tokens_per_step_pipelined(r.k, wl["match"]) if r.pipe else
                                          expected_tokens_per_step(r.k, wl["match"], branch_matches(wl)), 4),
        "steps_per_generation": steps_per_gen,
        "step_hbm": {"bytes": int(step_bytes), "achieved_gbs": round(step_gbs, 1),
                     "frac_of_8tbs": round(step_gbs / NOMINAL_HBM_GBS, 4),
                     "frac_of_measured": round(step_gbs / peak, 4)},
        "roofline": {"kernel": "gemm_kernel, gate/up launch (K %d, N %d, M %s)" %
                               (shape.d_model, 2 * shape.ffn_dim, "/".join(str(m) for m in sorted({r.b * r.q, r.b * r.q2}))),
                     "bound": "hbm", "achieved": round(gu_achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(gu_achieved / peak, 4),
                     "traffic": int(GEMM_TRAFFIC_RATIO * gu_bytes) if GEMM_TRAFFIC_CURRENT else None,
                     "traffic_source": GEMM_TRAFFIC_SOURCE, "peak_source": peak_kind,
                     "bytes_per_launch": int(gu_bytes), "ms_per_launch": round(gu_ms / max(1, gu_n), 5),
                     "launches": gu_n, "share_of_profiled_step": round(gu_ms / max(1e-9, prof_ms), 4),
                     "timing": "profiled pass: CUDA events around every launch on the context stream, so launches "
                               "are serialised (no programmatic dependent launch overlap): %.3f ms per step there "
                               "against %.3f ms graph-replayed; per-kernel fractions are lower bounds" %
                               (prof_ms / n_prof, ms_step),
                     "all_gemm": {"achieved": round(achieved, 1), "frac": round(achieved / peak, 4),
                                  "launches": g_launches, "bytes_per_launch": int(g_bytes / max(1, g_launches)),
                                  "ms_per_launch": round(g_ms / max(1, g_launches), 5)}},
        "kernels": {k: {"launches": v[0], "ms_total": round(v[1], 4), "us_per_launch": round(1e3 * v[1] / v[0], 2)}
                    for k, v in kstats.items()},
        "e2e": e2e, "gpu_launches": gpu_launches, "device_error_flags": flags,
        "prefill": prefill_line(r),
    }
    if r.pipe:
        out["config"].update({"pipelined": True, "note": "pipelined variant (not a step of the paper): every "
                              "block is [y, k drafts, k adaptive tokens]; one forward per step"})
    if r.tree:
        out["config"].update({"tree_width": r.width, "q2": r.q2,
                              "tree": "width chains of k drafts below the root (Sec. 2.1.2)"})
    if clk:
        out["clocks"] = clk
    return r, out


def prefill_line(r, chunk=512):
    """The prompt prefill (not part of the timed decode steps): tokens/s and its tensor-core
    rate.  FLOPs = 2 x positions x decoder-layer weights (the projections) + the causal
    attention products 2 x 2 x n^2/2 x H x hd per layer (algorithmic; the hi + lo operand
    split doubles what the tensor cores execute for the projections)."""
    n = r.P - 1
    sec = r.prefill_ms / 1e3
    sh = r.shape
    layer_w = sh.n_layers * (4 * sh.n_heads * sh.head_dim * sh.d_model + 3 * sh.ffn_dim * sh.d_model)
    flops = 2.0 * n * layer_w + sh.n_layers * 2.0 * 2.0 * (n * n / 2.0) * sh.n_heads * sh.head_dim
    tpk, kind = tensor_peak()
    tf = flops / sec / 1e12
    return {"tokens": n, "ms": round(r.prefill_ms, 3), "tokens_per_s": round(n / sec, 1), "chunk_rows": chunk,
            "tflops": round(tf, 1), "frac_of_measured_bf16": round(tf / tpk, 4), "peak": tpk, "peak_source": kind,
            "note": "tiled tcgen05 GEMM (128 weight rows x 128 positions), causal flash attention over "
                    "64-position blocks"}


def step_calls(r):
    """The C-ABI calls of one step once its block input is in place, by step kind (1: draft
    step 1; 2: draft step 2 or the tree step; the pipelined variant has one kind)."""
    wl = r.wl
    if r.pipe:
        def pipe():
            r.ctx.block_forward(r.kv, r.toks, r.logits, r.b, r.q)
            r.ctx.accept_pipelined(r.kv, r.logits, r.toks, r.pnver, r.b, r.q, r.acc, r.out,
                                   temperature=wl["temperature"], top_p=wl["top_p"], seed=1234, top_k=wl["top_k"])
        return {1: pipe}

    def step1():
        r.ctx.block_forward(r.kv, r.toks, r.logits, r.b, r.q)
        r.accept(0)

    def step2():
        if r.tree:
            r.forward_accept_tree()
        else:
            r.ctx.block_forward(r.kv, r.toks, r.logits, r.b, r.q)
            r.accept(r.k)
    return {1: step1, 2: step2}


def graph_calls(r, calls):
    """The same calls as CUDA graphs (one replay per step), or the eager calls if capture fails."""
    torch = r.torch
    try:
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            for f in calls.values():
                f()
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        out = {}
        for key, f in calls.items():
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                f()
            out[key] = g.replay
        torch.cuda.synchronize()
        return out, "CUDA graph of the step's C-ABI calls"
    except Exception as e:  # graphs are an optimisation; the eager calls run the same kernels
        print("note: e2e graph capture failed (%s); eager calls" % e, file=sys.stderr)
        torch.cuda.synchronize()
        return calls, "eager C-ABI calls"


def run_e2e(r, steps, steps_per_gen):
    """The decode loop a host program writes against the C ABI: every step the host builds
    the block input from the previous step's emitted tokens (pinned buffer -> device copy),
    runs the step's calls (block_forward and accept; a tree step: the tree forward and tree
    accept) as one CUDA-graph replay, copies the emitted tokens and accepted lengths back and
    reads them before the next step."""
    import numpy as np
    import torch
    b, k = r.b, r.k
    qm = r.qmax
    tok_h = torch.zeros(b * qm, dtype=torch.int32).pin_memory()
    out_h = torch.zeros(b * qm, dtype=torch.int32).pin_memory()
    acc_h = torch.zeros(b, dtype=torch.int32).pin_memory()
    table = r.table.cpu()
    adaptive = [r.shape.adaptive_id] * k
    fns, how = graph_calls(r, step_calls(r))
    r.reset()
    torch.cuda.synchronize()

    def start():
        return [r.P - 1] * b, [[int(r.prompts[s][-1])] for s in range(b)], [1] * b

    lens, last_out, last_acc = start()
    tokens = 0
    h2d = d2h = 0
    st = torch.cuda.current_stream()
    if r.pipe:
        return run_e2e_pipelined(r, steps, steps_per_gen, tok_h, out_h, acc_h, table, adaptive, start, fns[1], how)
    # the host side works on numpy views of the pinned buffers (no per-step allocations)
    tok_np, out_np, acc_np = tok_h.numpy(), out_h.numpy(), acc_h.numpy()
    table_np = table.numpy()
    adaptive_np = np.asarray(adaptive, dtype=np.int32)
    t0 = time.perf_counter()
    for i in range(steps):
        j = i % steps_per_gen
        if j == 0 and i > 0:
            r.reset()
            lens, last_out, last_acc = start()
        mode = 1 if j % 2 == 0 else 2
        q = r.q if mode == 1 else r.q2
        for s in range(b):
            if mode == 1:
                tok_np[s * q] = last_out[s][last_acc[s] - 1]
                tok_np[s * q + 1:s * q + q] = adaptive_np
            else:
                tok_np[s * q] = last_out[s][0]
                for w in range(r.width):
                    tok_np[s * q + 1 + w * k:s * q + 1 + (w + 1) * k] = table_np[w, s, lens[s] + 1:lens[s] + k + 1]
        r.toks[:b * q].copy_(tok_h[:b * q], non_blocking=True)
        fns[mode]()
        out_h[:b * q].copy_(r.out[:b * q], non_blocking=True)
        acc_h.copy_(r.acc, non_blocking=True)
        st.synchronize()
        for s in range(b):
            last_out[s] = out_np[s * q:(s + 1) * q].copy()
            last_acc[s] = int(acc_np[s])
            lens[s] += last_acc[s]
        tokens += int(acc_np.sum())
        h2d += b * q * 4
        d2h += b * q * 4 + b * 4
    t1 = time.perf_counter()
    return {"value": round(tokens / (t1 - t0), 2), "unit": "tokens/s", "h2d_bytes_per_step": round(h2d / steps, 1),
            "d2h_bytes_per_step": round(d2h / steps, 1), "launch": how + ", host sync each step"}


def run_e2e_pipelined(r, steps, steps_per_gen, tok_h, out_h, acc_h, table, adaptive, start, fn, how):
    """run_e2e for the pipelined variant: the host keeps each sequence's block mode, builds
    [x_0, drafts or adaptive ids, adaptive ids] and copies the per-sequence verify counts in."""
    import numpy as np
    import torch
    b, k, q = r.b, r.k, r.q
    nv_h = torch.zeros(b, dtype=torch.int32).pin_memory()
    # the host side works on numpy views of the pinned buffers (no per-step allocations)
    tok_np, out_np, acc_np, nv_np = tok_h.numpy(), out_h.numpy(), acc_h.numpy(), nv_h.numpy()
    table_np = table.numpy()
    adaptive_np = np.asarray(adaptive, dtype=np.int32)
    lens, last_out, last_acc = start()
    prev_mode = [1] * b
    tokens = h2d = d2h = 0
    st = torch.cuda.current_stream()
    t0 = time.perf_counter()
    for i in range(steps):
        if i % steps_per_gen == 0 and i > 0:
            r.reset()
            lens, last_out, last_acc = start()
            prev_mode = [1] * b
        for s in range(b):
            a_mode = prev_mode[s] == 0 or last_acc[s] == k + 1
            tok_np[s * q] = last_out[s][last_acc[s] - 1]
            tok_np[s * q + 1:s * q + 1 + k] = table_np[0, s, lens[s] + 1:lens[s] + k + 1] if a_mode else adaptive_np
            tok_np[s * q + 1 + k:s * q + 1 + 2 * k] = adaptive_np
            nv_np[s] = k if a_mode else 0
            prev_mode[s] = 1 if a_mode else 0
        r.toks[:b * q].copy_(tok_h[:b * q], non_blocking=True)
        r.pnver.copy_(nv_h, non_blocking=True)
        fn()
        out_h[:b * q].copy_(r.out[:b * q], non_blocking=True)
        acc_h.copy_(r.acc, non_blocking=True)
        st.synchronize()
        for s in range(b):
            last_out[s] = out_np[s * q:(s + 1) * q].copy()
            last_acc[s] = int(acc_np[s])
            lens[s] += last_acc[s]
        tokens += int(acc_np.sum())
        h2d += b * q * 4 + b * 4
        d2h += b * q * 4 + b * 4
    t1 = time.perf_counter()
    return {"value": round(tokens / (t1 - t0), 2), "unit": "tokens/s", "h2d_bytes_per_step": round(h2d / steps, 1),
            "d2h_bytes_per_step": round(d2h / steps, 1), "launch": how + ", host sync each step"}


# ----------------------------------------------------------------------------- CPU oracle
def oracle_sample(shape_name, wl, weights_gpu=None, n_layers=2, repeat=1, gen_device="cpu"):
    """Time the CPU oracle on a bounded sample of one block step at the workload's shape:
    `n_layers` decoder layers (their weights widened once and cached, as the oracle does)
    against a synthetic KV of the prompt length, plus the final norm + LM head, then
    extrapolate to all layers.  Returns (seconds per full step, details)."""
    import numpy as np
    import torch
    import synth
    from oracle import model as OM
    shape = synth.SHAPES[shape_name]
    q = mean_rows(wl)
    P = wl["prompt"]

    def provider(name, layer):
        if weights_gpu is not None:
            t = weights_gpu[name] if layer < 0 else weights_gpu["layers"][layer][name]
            return t.cpu()
        return synth.make_weight(shape, name, layer, wl.get("seed", 0), "cpu")

    W = OM.Weights(shape, provider=provider, cache=True)
    small = synth.ModelShape("sample", n_layers, shape.d_model, shape.n_heads, shape.head_dim, shape.ffn_dim,
                             shape.vocab, shape.adaptive_id)
    kv = OM.KVCache(small, 1, P + q)
    for l in range(n_layers):
        for which, dst in ((0, kv.K), (1, kv.V)):
            vals = synth.kv_values(0, l, which, (shape.n_heads, P, shape.head_dim), device=gen_device)
            dst[l][0][:, :P] = vals.cpu().double().numpy()
    kv.len[0] = P
    toks = synth.uniform_ids(0, 999, q, shape.adaptive_id).tolist()
    # widen the sampled weights once (the oracle caches them)
    for l in range(n_layers):
        for n in synth.LAYER_MATS:
            W.get(n, l)
    for n in ("embed", "final_norm", "lm_head"):
        W.get(n)
    t0 = time.perf_counter()
    for _ in range(repeat):
        OM.block_forward(W, kv, 0, toks, layers=range(n_layers), final=False)
    t_layers = (time.perf_counter() - t0) / repeat
    t0 = time.perf_counter()
    OM.block_forward(W, kv, 0, toks, layers=[], final=True)
    t_head = time.perf_counter() - t0
    per_layer = t_layers / n_layers
    return shape.n_layers * per_layer + t_head, {"per_layer_s": per_layer, "head_s": t_head}


def mean_rows(wl):
    """Block rows of the workload's average step (steps alternate k + 1 and 1 + width * k rows;
    pipelined blocks have 2k + 1)."""
    if wl.get("pipelined"):
        return 2 * wl["k"] + 1
    return round((wl["k"] + 1 + 1 + wl.get("width", 1) * wl["k"]) / 2)


def workload_tokens_per_step(wl):
    """The stub's expected tokens per block step for the workload."""
    if wl.get("pipelined"):
        return expected_tokens_per_step_pipelined(wl["k"], wl["match"])
    return expected_tokens_per_step(wl["k"], wl["match"], branch_matches(wl))


def cpu_baseline(args, wl, weights_gpu):
    tps = workload_tokens_per_step(wl)
    dev = next(iter(weights_gpu["layers"][0].values())).device if weights_gpu is not None else "cpu"
    t_step, det = oracle_sample(wl["shape"], wl, weights_gpu, n_layers=2, gen_device=dev)
    return {"value": round(tps / t_step, 4), "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": ("one q=%d block step at context %d: 2 of %d decoder layers timed (weights widened and cached "
                       "first) plus the final norm + LM head, extrapolated to all layers (%.2f s/layer, %.2f s head); "
                       "tokens/step = %.3f, the stub's expectation" %
                       (mean_rows(wl), wl["prompt"], __import__("synth").SHAPES[wl["shape"]].n_layers,
                        det["per_layer_s"], det["head_s"], tps)),
            "s_per_step": round(t_step, 3)}


def run_reference(args, wl, rank, world):
    """The reference arm: the CPU oracle (no reference implementation exists).  Each step is a
    bounded sample -- one decoder layer of the block step -- scaled by the layer count."""
    import synth
    from oracle import model as OM
    shape = synth.SHAPES[wl["shape"]]
    tps = workload_tokens_per_step(wl)
    q = mean_rows(wl)
    P = wl["prompt"]
    W = OM.Weights(shape, provider=lambda n, l: synth.make_weight(shape, n, l, wl.get("seed", 0), "cpu"), cache=True)
    small = synth.ModelShape("sample", 1, shape.d_model, shape.n_heads, shape.head_dim, shape.ffn_dim,
                             shape.vocab, shape.adaptive_id)
    kv = OM.KVCache(small, 1, P + q)
    kv.K[0][0][:, :P] = synth.kv_values(0, 0, 0, (shape.n_heads, P, shape.head_dim)).double().numpy()
    kv.V[0][0][:, :P] = synth.kv_values(0, 0, 1, (shape.n_heads, P, shape.head_dim)).double().numpy()
    kv.len[0] = P
    toks = synth.uniform_ids(0, 999, q, shape.adaptive_id).tolist()
    for n in synth.LAYER_MATS:
        W.get(n, 0)
    for n in ("embed", "final_norm", "lm_head"):
        W.get(n)
    t0 = time.perf_counter()
    OM.block_forward(W, kv, 0, toks, layers=[], final=True)
    t_head = time.perf_counter() - t0
    for _ in range(args.warmup):
        OM.block_forward(W, kv, 0, toks, layers=[0], final=False)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        OM.block_forward(W, kv, 0, toks, layers=[0], final=False)
        times.append(time.perf_counter() - t0)
    per_layer = statistics.mean(times)
    # one whole block step of one sequence, extrapolated; a batch of b sequences takes b times as
    # long on the oracle (it runs the sequences one after another), so tokens/s do not depend on b
    t_full = shape.n_layers * per_layer + t_head
    value = tps / t_full
    sample = ("each timed step is one decoder layer of a q=%d block step at context %d (weights widened once and "
              "cached); a whole block step is extrapolated as %d layers plus the final norm + LM head timed once "
              "(%.2f s); tokens/step = %.3f per sequence, the stub's expectation" %
              (q, P, shape.n_layers, t_head, tps))
    return {"metric": METRIC, "value": round(value, 4), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(per_layer * 1e3, 2), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": args.config, "model": shape.name + "-shaped random init (seed %d)" % wl.get("seed", 0),
                       "global_batch": wl["batch"], "seq_len": P, "k": wl["k"]},
            "sample_step": "one decoder layer of the block step (the elapsed time of each timed step is ms_per_step)",
            "extrapolated_ms_per_block_step": round(t_full * 1e3, 2),
            "tokens_per_step_basis": "the draft stub's expected tokens per block step (%.4f per sequence); the GPU "
                                     "arm reports the same basis as value_expected_basis" % tps,
            "cpu_baseline": {"value": round(value, 4), "unit": "tokens/s", "cores": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


# ----------------------------------------------------------------------------- kernel sweeps
SWEEP_GEMM_SHAPES = [(4096, 12288), (4096, 22016), (11008, 4096), (4096, 32016)]   # (K, N): QKV, gate+up, down, head
SWEEP_Q = [1, 2, 4, 6, 8, 11, 16]
SWEEP_CTX = [512, 2048, 8192, 16384]


def run_ksweep(args):
    """k-sweep (one JSON line per k): block step time, tokens per step, accept rate and
    tokens/s of the workload's generation loop for k adaptive tokens (q = k + 1), the same
    weights throughout.  Checks that the step time stays almost flat in k (Sec. 3.4.1)."""
    import torch
    import synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    base = dict(WORKLOADS[args.config])
    ks = [int(v) for v in args.ks.split(",")] if args.ks else list(range(1, 14))
    weights = synth.make_model(synth.SHAPES[base["shape"]], seed=0, device=dev)
    for k in ks:
        wl = dict(base, k=k)
        r = Runner(wl, dev, weights=weights)
        steps_per_gen, lens, toks_cal, flags = r.calibrate()
        graphs = r.capture()
        r.reset()
        r.run_steps(4, steps_per_gen, graphs)
        r.reset()
        n = steps_per_gen
        em0 = r.ctx.kv_emitted(r.kv).sum().item()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        r.run_steps(n, steps_per_gen, graphs)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        tokens = r.ctx.kv_emitted(r.kv).sum().item() - em0
        print(json.dumps({"kind": "ksweep", "workload": args.config, "k": k, "q": k + 1, "q2": r.q2, "steps": n,
                          "ms_per_step": round(ms / n, 4), "tokens_per_step": round(tokens / r.b / n, 4),
                          "expected_tokens_per_step": round(expected_tokens_per_step(k, wl["match"], branch_matches(wl)), 4),
                          "accept_rate": accept_rate(r, toks_cal), "tokens_per_s": round(tokens / (ms / 1e3), 2),
                          "device_error_flags": flags | r.ctx.get_error()}), flush=True)
        del graphs, r
        torch.cuda.synchronize()


def kernel_us(ctx, name, reps, call):
    """Mean device time of one launch of kernel class `name` over `reps` calls, from the
    library's profiling hook (CUDA events around each launch)."""
    ctx.profile_begin(2 * reps + 16)
    for i in range(reps):
        call(i)
    st = ctx.profile_end()
    n, ms = st.get(name, (0, 0.0))
    return 1e3 * ms / n if n else float("nan")


def run_sweep(args):
    """Kernel sweeps on 7B shapes (one JSON line per case): the skinny GEMM with M = q against
    bf16 weights, and block-causal attention of q rows (32 heads x 128) against a bf16 cache.
    Weights/caches rotate over enough buffers to exceed L2 between repetitions."""
    import torch
    import synth
    import paper_2403_18647_gb300 as sd
    torch.cuda.set_device(0)
    peak, kind = peaks()
    ctx = sd.Context(synth.SHAPES["7b"], None, max_position=16384 + 64)
    reps = args.reps
    l2 = torch.cuda.get_device_properties(0).L2_cache_size
    cases = []
    if args.sweep in ("gemm", "all"):
        shapes = [tuple(int(v) for v in args.shape.split("x"))] if args.shape else SWEEP_GEMM_SHAPES
        qs = [args.m] if args.m else SWEEP_Q
        for K, N in shapes:
            nbuf = max(2, int(math.ceil(4 * l2 / (K * N * 2))))
            ws = [synth.normal_bf16(7, i, (N, K), 0.02, device="cuda") for i in range(nbuf)]
            for M in qs:
                x = synth.normal_f32(7, 100 + M, (M, K), 1.0, device="cuda")
                y = torch.empty(M, N, device="cuda")
                for i in range(3):
                    ctx.op_gemm(x, ws[i % nbuf], y)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record()
                for i in range(reps):
                    ctx.op_gemm(x, ws[i % nbuf], y)
                e1.record()
                torch.cuda.synchronize()
                us = e0.elapsed_time(e1) * 1e3 / reps
                kus = kernel_us(ctx, "gemm_op", reps, lambda i: ctx.op_gemm(x, ws[i % nbuf], y))
                by = K * N * 2 + M * K * 4 + M * N * 4
                cases.append({"kernel": "skinny_gemm", "M": M, "K": K, "N": N, "us": round(us, 2),
                              "GB/s": round(by / us / 1e3, 1), "frac_of_measured": round(by / us / 1e3 / peak, 4),
                              "frac_of_8tbs": round(by / us / 1e3 / NOMINAL_HBM_GBS, 4),
                              "kernel_us": round(kus, 2), "kernel_GB/s": round(by / kus / 1e3, 1),
                              "kernel_frac_of_measured": round(by / kus / 1e3 / peak, 4),
                              "note": "us: back-to-back calls, each with the fp32 -> bf16 hi/lo operand split kernel; "
                                      "kernel_us: the GEMM kernel alone (CUDA events around each launch)"})
            del ws
    if args.sweep in ("attention", "all"):
        H, hd = 32, 128
        ctxs = [args.ctx] if args.ctx else SWEEP_CTX
        qs = [args.m] if args.m else SWEEP_Q
        for n in ctxs:
            cap = n + 16
            nbuf = max(2, int(math.ceil(4 * l2 / (2 * H * cap * hd * 2))))
            Ks = [synth.normal_bf16(8, 2 * i, (H * cap, hd), 1.0, device="cuda") for i in range(nbuf)]
            Vs = [synth.normal_bf16(8, 2 * i + 1, (H * cap, hd), 1.0, device="cuda") for i in range(nbuf)]
            ln = torch.tensor([n], dtype=torch.int32, device="cuda")
            for q in qs:
                Q = synth.normal_f32(8, 50 + q, (q, H * hd), 1.0, device="cuda")
                out = torch.empty(q, H * hd, device="cuda")
                for i in range(3):
                    ctx.op_attention(Q, Ks[i % nbuf], Vs[i % nbuf], ln, 1, q, H, hd, cap, out)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record()
                for i in range(reps):
                    ctx.op_attention(Q, Ks[i % nbuf], Vs[i % nbuf], ln, 1, q, H, hd, cap, out)
                e1.record()
                torch.cuda.synchronize()
                us = e0.elapsed_time(e1) * 1e3 / reps
                kus = kernel_us(ctx, "attention_op", reps,
                                lambda i: ctx.op_attention(Q, Ks[i % nbuf], Vs[i % nbuf], ln, 1, q, H, hd, cap, out))
                by = 2 * H * (n + q) * hd * 2 + 2 * q * H * hd * 4
                cases.append({"kernel": "attention", "q": q, "ctx": n, "heads": H, "head_dim": hd,
                              "us": round(us, 2), "GB/s": round(by / us / 1e3, 1),
                              "frac_of_measured": round(by / us / 1e3 / peak, 4),
                              "frac_of_8tbs": round(by / us / 1e3 / NOMINAL_HBM_GBS, 4),
                              "kernel_us": round(kus, 2), "kernel_GB/s": round(by / kus / 1e3, 1),
                              "kernel_frac_of_measured": round(by / kus / 1e3 / peak, 4)})
            del Ks, Vs
    if args.sweep in ("prefill", "all"):
        # the prefill path's tiled GEMM (M positions x the 7B projections), tensor-core bound
        tpk, tkind = tensor_peak()
        shapes = [tuple(int(v) for v in args.shape.split("x"))] if args.shape else SWEEP_GEMM_SHAPES[:3]
        ms = [args.m] if args.m else [128, 256, 512]
        for K, N in shapes:
            w = synth.normal_bf16(9, 1, (N, K), 0.02, device="cuda")
            for M in ms:
                x = synth.normal_f32(9, 100 + M, (M, K), 1.0, device="cuda")
                y = torch.empty(M, N, device="cuda")
                for i in range(3):
                    ctx.op_gemm(x, w, y)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record()
                for i in range(reps):
                    ctx.op_gemm(x, w, y)
                e1.record()
                torch.cuda.synchronize()
                us = e0.elapsed_time(e1) * 1e3 / reps
                alg = 2.0 * M * N * K / us / 1e6          # TFLOP/s of y = x W^T
                cases.append({"kernel": "prefill_gemm", "M": M, "K": K, "N": N, "us": round(us, 2),
                              "TFLOP/s": round(alg, 1), "frac_of_measured_bf16": round(alg / tpk, 4),
                              "tensor_TFLOP/s": round(2 * alg, 1), "tensor_frac": round(2 * alg / tpk, 4),
                              "peak": tpk, "peak_source": tkind,
                              "note": "x enters as bf16 hi + lo: the tensor cores execute 2 x 2MNK; includes "
                                      "the fp32 -> bf16 hi/lo operand split kernel"})
            del w
        # a whole prefill at 7B layer dimensions (two layers, so that a profiler capture holds
        # under a GB): per-kernel device time, and the causal attention's rate
        sh7 = synth.SHAPES["7b"]
        sh = synth.ModelShape("7b-2layers", 2, sh7.d_model, sh7.n_heads, sh7.head_dim, sh7.ffn_dim, sh7.vocab,
                              sh7.adaptive_id)
        n = args.ctx if args.ctx else 2047
        wts = synth.make_model(sh, seed=0, device="cuda")
        pctx = sd.Context(sh, wts, max_position=n + 64)
        kv = pctx.kv(1, n + 16)
        prompt = synth.prompt_ids(0, 0, n, sh.adaptive_id).cuda()
        zero = torch.zeros(1, dtype=torch.int32, device="cuda")
        for _ in range(2):
            pctx.kv_commit(kv, zero, 1)
            pctx.prefill(kv, 0, prompt)
        torch.cuda.synchronize()
        pctx.kv_commit(kv, zero, 1)
        pctx.profile_begin(4096)
        pctx.prefill(kv, 0, prompt)
        st = pctx.profile_end()
        att = st.get("prefill_attention", (0, 0.0))
        att_flops = sh.n_layers * 2.0 * 2.0 * (n * n / 2.0) * sh.n_heads * sh.head_dim
        cases.append({"kernel": "prefill_step", "shape": sh.name, "positions": n,
                      "kernels_ms": {k: round(v[1], 4) for k, v in st.items()},
                      "attention_TFLOP/s": round(att_flops / (att[1] / 1e3) / 1e12, 1) if att[1] else None,
                      "note": "launches timed one by one (CUDA events); attention FLOPs 4 x n^2/2 x H x hd per "
                              "layer (causal), algorithmic"})
        del pctx, kv, wts
    for c in cases:
        print(json.dumps(c), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="7b", choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", choices=["gemm", "attention", "prefill", "all"],
                    help="kernel sweeps instead of the step bench")
    ap.add_argument("--shape", default="", help="sweep one GEMM shape KxN")
    ap.add_argument("--m", type=int, default=0, help="sweep one M (GEMM) or q (attention)")
    ap.add_argument("--ctx", type=int, default=0, help="sweep one attention context length")
    ap.add_argument("--reps", type=int, default=50)
    ap.add_argument("--ksweep", action="store_true", help="k-sweep of the generation loop (k = 1..13)")
    ap.add_argument("--ks", default="", help="k values for --ksweep, comma separated")
    ap.add_argument("--k", type=int, default=None, help="adaptive tokens per block (overrides the workload's)")
    ap.add_argument("--new-tokens", type=int, default=None, help="tokens generated per generation")
    ap.add_argument("--seed", type=int, default=None, help="seed of the synthetic weights")
    args = ap.parse_args()
    if args.sweep:
        run_sweep(args)
        return
    if args.ksweep:
        run_ksweep(args)
        return
    if args.warmup < 3:
        args.warmup = 3
    wl = dict(WORKLOADS[args.config])
    for key, val in (("k", args.k), ("new", args.new_tokens), ("seed", args.seed)):
        if val is not None:
            wl[key] = val
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, wl, rank, world)), flush=True)
        return
    import torch
    import torch.distributed as dist
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0"))))
    r, out = run_ours(args, wl, rank, world)
    if rank == 0:
        if not args.no_cpu_baseline:
            try:
                out["cpu_baseline"] = cpu_baseline(args, wl, r.weights)
            except Exception as e:  # keep the GPU line even if the host runs out of memory
                out["cpu_baseline"] = {"value": None, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                                       "sample": "failed: %s" % e}
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
