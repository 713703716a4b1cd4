#!/usr/bin/env python
"""Mixed-iteration benchmark on GB300: prints ONE JSON line.

Workload (default, the headline): Qwen3-32B attention geometry (64 Q / 8 KV
heads, head dim 128, bf16, 16-token pages), 64 layer calls per iteration with
distinct per-layer pools (~200 GB in all), 128 decodes with cached contexts
log-uniform in [1024, 16384], and one 32768-token prompt prefilled beside them
with chunk size p swept over {0, 1024, 2048, 4096, 8192}, every chunk in order
(61 iterations).  One step = that whole sweep.  Inputs are seeded synthetic
N(0,1) bf16 values, resident in HBM before timing; the pools are far larger
than L2.  The Qwen3-0.6B (28 layers) and Qwen3-8B (36 layers) sweeps are
measured in the same run and reported beside it (`other_configs`).

`value` = tokens (decode tokens + prompt tokens) per second of device time,
from CUDA events on the launching stream; `e2e` = the same through the C-ABI
iteration call with host buffers (q/k/v copied in from pinned host memory and
outputs copied out inside the timed region).  `--impl reference` times the
float64 CPU oracle on a bounded sample instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

SPEC_HBM = 8000e9          # nominal HBM3e bytes/s
SPEC_TFLOPS = 1706.7e12   # nominal sustained dense bf16 flop/s
METRIC = ("mixed-iteration device µs & tokens/s; % of HBM/tensor roofline per chunk size")
UNIT = "tokens/s"
DEFAULT_CONFIG = "qwen3-32b-attn-64L-chunk-sweep"
# sweeps reported beside the headline in the same run
SIDE_CONFIGS = ("qwen3-0.6b-attn-28L-chunk-sweep", "qwen3-8b-attn-36L-chunk-sweep")
# sweeps whose per-iteration inputs for every layer would not fit beside the
# pools: one q/k/v buffer per layer, reused by every iteration
LEAN_CONFIGS = ("qwen3-32b-attn-64L-chunk-sweep",)
KERNEL_SRC = os.path.join(ROOT, "paper_2609_38386_gb300", "csrc", "mx_layer.cu")
# the committed ncu summary that gives each sweep's DRAM bytes per launch
TRAFFIC_SUMMARY = {
    "qwen3-0.6b-attn-28L-chunk-sweep": os.path.join(ROOT, "profiles", "mixed_layer_qwen06b_sweep.md"),
    "qwen3-32b-attn-64L-chunk-sweep": os.path.join(ROOT, "profiles", "mixed_layer_qwen32b_sweep.md"),
}


# ----------------------------------------------------------------- helpers
def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def kernel_hash():
    h = hashlib.sha256()
    for f in (KERNEL_SRC, os.path.join(ROOT, "paper_2609_38386_gb300", "csrc", "mx_ptx.cuh"),
              os.path.join(ROOT, "paper_2609_38386_gb300", "csrc", "mx_internal.h")):
        h.update(open(f, "rb").read())
    return h.hexdigest()[:16]


def committed_traffic(config):
    """DRAM bytes per launch of the sweep from its committed ncu summary, if
    that was taken on the current kernel source (else None)."""
    path = TRAFFIC_SUMMARY.get(config)
    if not path or not os.path.exists(path):
        return None
    txt = open(path).read()
    m_h = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", txt)
    m_t = re.search(r"dram_bytes_per_launch_full_workload:\s*([0-9.eE+]+)", txt)
    if not m_h or not m_t or m_h.group(1) != kernel_hash():
        return None
    return float(m_t.group(1))


class ClockSampler:
    """nvidia-smi clock/throttle samples during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = os.path.join("/tmp", f"mx_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", self.gpu_id], stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], [], set()
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for name, val in zip(self.NAMES, f[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        os.unlink(self.path)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


# Multi-GPU: independent replicas (the path partitions by request; no
# exchange inside attention).  Each rank runs the whole workload on its own
# GPU with its own seed; the job's time is the slowest rank's and its value
# the tokens of all ranks over that time.
def replica_seed_offset(rank: int) -> int:
    return rank


def max_over_ranks(value: float, ws: int, device=None) -> float:
    if ws == 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(tokens_per_step: int, steps: int, ws: int, total_ms: float) -> float:
    return tokens_per_step * steps * ws / (total_ms * 1e-3)


# ------------------------------------------------------------ GPU workload
class Workload:
    """Device-resident inputs of every iteration of a sweep, per layer."""

    def __init__(self, cfg, device, seed_offset=0, layers=None, lean=False):
        import torch

        import synth
        from paper_2609_38386_gb300 import Context
        from synth import device as sdev
        from synth import workload as wl

        self.cfg = cfg
        self.geom = g = cfg.geom
        self.L = layers or cfg.n_layers
        self.layout = lay = cfg.layout()
        self.its = cfg.iterations()
        self.seed = cfg.seed + seed_offset
        self.max_tok = max(it.n_tokens for it in self.its)
        self.ctx = Context(num_q_heads=g.hq, num_kv_heads=g.hkv, num_pages=lay.num_pages,
                           num_seqs=lay.num_seqs, max_pages_per_seq=lay.max_pages,
                           max_tokens=self.max_tok, max_decodes=max(cfg.n_decodes, 1),
                           device=device.index or 0)
        self.page_table = torch.from_numpy(lay.page_table).to(device)
        self.pools = []
        for l in range(self.L):
            kp = torch.empty(lay.pool_shape(), dtype=torch.int16, device=device)
            vp = torch.empty(lay.pool_shape(), dtype=torch.int16, device=device)
            sdev.fill_(kp, wl.pool_base(self.seed, l, synth.STREAM_KPOOL))
            sdev.fill_(vp, wl.pool_base(self.seed, l, synth.STREAM_VPOOL))
            self.pools.append((kp, vp))
        self.outs = [torch.empty((self.max_tok, g.hq, g.head_dim), dtype=torch.int16,
                                 device=device) for _ in range(self.L)]
        self.descs, self.layer_arrays, self.inputs, self.slots = [], [], [], []
        shared = []
        if lean:
            # one q/k/v buffer per layer, sized for the largest iteration and
            # reused by every iteration: for sweeps whose per-iteration inputs
            # do not fit (the 32B sweep would need ~225 GB of them)
            big = max(self.its, key=lambda it: it.n_tokens)
            for l in range(self.L):
                q = torch.empty((self.max_tok, g.hq, g.head_dim), dtype=torch.int16, device=device)
                k = torch.empty((self.max_tok, g.hkv, g.head_dim), dtype=torch.int16, device=device)
                v = torch.empty_like(k)
                sdev.fill_tokens_(q, self.seed, l, synth.STREAM_Q, big)
                sdev.fill_tokens_(k, self.seed, l, synth.STREAM_K, big)
                sdev.fill_tokens_(v, self.seed, l, synth.STREAM_V, big)
                shared.append((q, k, v))
        for it in self.its:
            sl = torch.from_numpy(it.slots(lay)).to(device)
            self.slots.append(sl)
            bufs, keep = [], []
            for l in range(self.L):
                if lean:
                    q, k, v = shared[l]
                else:
                    q = torch.empty((it.n_tokens, g.hq, g.head_dim), dtype=torch.int16,
                                    device=device)
                    k = torch.empty((it.n_tokens, g.hkv, g.head_dim), dtype=torch.int16,
                                    device=device)
                    v = torch.empty_like(k)
                    sdev.fill_tokens_(q, self.seed, l, synth.STREAM_Q, it)
                    sdev.fill_tokens_(k, self.seed, l, synth.STREAM_K, it)
                    sdev.fill_tokens_(v, self.seed, l, synth.STREAM_V, it)
                keep.append((q, k, v))
                kp, vp = self.pools[l]
                bufs.append(self.ctx.make_bufs(q, k, v, kp, vp, self.outs[l]))
            self.inputs.append(keep)
            self.layer_arrays.append(self.ctx.layer_array(bufs))
            self.descs.append(self.ctx.make_desc(
                decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
                prefill_seq_id=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t,
                page_table=self.page_table, slots=sl))
        torch.cuda.synchronize(device)
        self.work = [wl.algorithmic_work(g, it) for it in self.its]
        self.tokens_per_step = sum(it.n_tokens for it in self.its)

    def close(self):
        """Release the context and the device tensors."""
        self.ctx.close()
        self.pools = self.outs = self.inputs = self.slots = None
        self.descs = self.layer_arrays = None

    def run_step(self, events=None):
        """Enqueue every iteration of the sweep (no host waits)."""
        for i in range(len(self.its)):
            if events is not None:
                events[i].record()
            self.ctx.iteration(self.descs[i], self.layer_arrays[i], wait=False)
        if events is not None:
            events[len(self.its)].record()


def e2e_measure(w, steps, device, budget_bytes=12 << 30):
    """Same sweep through the iteration call with host buffers: every
    iteration's q/k/v for all layers is copied from pinned host memory, the
    iteration runs, and every layer's output is copied back to pinned host
    memory, all inside the timed region.  The copies are pipelined against
    the compute the way a serving loop would run them, in units of a group of
    consecutive layers (the whole iteration when its buffers fit the budget;
    for the 64-layer 32B sweep, whose pools fill most of HBM, 8 layers, each
    group one iteration call): the inputs of unit j+1 and j+2 upload on one
    stream and the outputs of unit j-1 download on another while unit j
    computes (three device buffer sets).  The pipeline runs across the timed
    steps; the region ends when the last step's outputs are on the host.  The
    host buffer holds the largest iteration's inputs; each unit uploads as
    many bytes as its own iteration needs (so the copy volume is exact, while
    the contents are those of the largest iteration)."""
    import torch
    g, L = w.geom, w.L
    per_tok_in = (g.hq + 2 * g.hkv) * g.head_dim
    per_tok_out = g.hq * g.head_dim
    nbuf = 3
    group = L
    for cand in range(1, L + 1):                     # fewest groups that fit
        if L % cand == 0 and nbuf * (L // cand) * w.max_tok * (per_tok_in + per_tok_out) * 2 <= budget_bytes:
            group = L // cand
            break
    else:
        group = 1
    n_groups = L // group
    max_in = group * w.max_tok * per_tok_in
    max_out = group * w.max_tok * per_tok_out
    h_in = torch.empty(max_in, dtype=torch.int16, pin_memory=True)
    h_out = torch.empty(max_out, dtype=torch.int16, pin_memory=True)
    d_in = [torch.empty(max_in, dtype=torch.int16, device=device) for _ in range(nbuf)]
    d_out = [torch.empty(max_out, dtype=torch.int16, device=device) for _ in range(nbuf)]
    # host contents: the largest iteration's device inputs of the first group
    big = max(range(len(w.its)), key=lambda i: w.its[i].n_tokens)
    nb = w.its[big].n_tokens
    off = 0
    for l in range(group):
        for t, heads in zip(w.inputs[big][l], (g.hq, g.hkv, g.hkv)):
            n = nb * heads * g.head_dim
            h_in[off:off + n].copy_(t.reshape(-1)[:n].cpu())
            off += n
    # per (iteration, layer group, buffer set): the layer array of that unit
    arrays, in_elems, out_elems = [], [], []
    for it in w.its:
        n = it.n_tokens
        per_group = []
        for gi in range(n_groups):
            sets = []
            for b in range(nbuf):
                bufs, o_in, o_out = [], 0, 0
                for l in range(gi * group, (gi + 1) * group):
                    q = d_in[b][o_in:o_in + n * g.hq * g.head_dim]
                    o_in += q.numel()
                    k = d_in[b][o_in:o_in + n * g.hkv * g.head_dim]
                    o_in += k.numel()
                    v = d_in[b][o_in:o_in + n * g.hkv * g.head_dim]
                    o_in += v.numel()
                    out = d_out[b][o_out:o_out + n * per_tok_out]
                    o_out += out.numel()
                    kp, vp = w.pools[l]
                    bufs.append(w.ctx.make_bufs(q, k, v, kp, vp, out))
                sets.append(w.ctx.layer_array(bufs))
            per_group.append(sets)
        arrays.append(per_group)
        in_elems.append(group * n * per_tok_in)
        out_elems.append(group * n * per_tok_out)
    comp = torch.cuda.current_stream(device)
    up = torch.cuda.Stream(device)
    down = torch.cuda.Stream(device)
    n_it = len(w.its)

    def run(n_steps):
        # one continuous pipeline over the steps' units: unit j uses buffer
        # set j % nbuf, uploads as soon as unit j - nbuf has consumed that
        # set, and downloads as soon as it has computed
        units = [(i, gi) for _ in range(n_steps) for i in range(n_it) for gi in range(n_groups)]
        total = len(units)
        ev_in = [torch.cuda.Event() for _ in range(total)]
        ev_comp = [torch.cuda.Event() for _ in range(total)]
        ev_out = [torch.cuda.Event() for _ in range(total)]
        for j, (i, gi) in enumerate(units):
            b = j % nbuf
            with torch.cuda.stream(up):
                if j >= nbuf:
                    up.wait_event(ev_comp[j - nbuf])   # inputs of j-nbuf consumed
                d_in[b][:in_elems[i]].copy_(h_in[:in_elems[i]], non_blocking=True)
                ev_in[j].record(up)
            comp.wait_event(ev_in[j])
            if j >= nbuf:
                comp.wait_event(ev_out[j - nbuf])      # outputs of j-nbuf downloaded
            w.ctx.iteration(w.descs[i], arrays[i][gi][b], stream=comp, wait=False)
            ev_comp[j].record(comp)
            with torch.cuda.stream(down):
                down.wait_event(ev_comp[j])
                h_out[:out_elems[i]].copy_(d_out[b][:out_elems[i]], non_blocking=True)
                ev_out[j].record(down)
        for s_ in (up, comp, down):
            s_.synchronize()

    run(1)  # warm-up
    w.ctx.sync_status()
    torch.cuda.synchronize(device)
    t0 = time.perf_counter()
    run(steps)
    torch.cuda.synchronize(device)
    dt = time.perf_counter() - t0
    w.ctx.sync_status()
    res = {"value": w.tokens_per_step * steps / dt, "unit": UNIT,
           "h2d_bytes_per_step": int(sum(in_elems) * 2 * n_groups),
           "d2h_bytes_per_step": int(sum(out_elems) * 2 * n_groups),
           "seconds": dt, "steps": steps, "layers_per_call": group,
           "copies": "pinned host <-> device on two copy streams, pipelined with compute across the "
                     "timed steps in units of %d layer(s) per iteration call (every step's inputs and "
                     "outputs inside the region); each unit copies its own iteration's byte count, "
                     "taken from a host buffer that holds the largest iteration's inputs" % group}
    del d_in, d_out, h_in, h_out
    torch.cuda.empty_cache()
    return res


def independent_layers_measure(w, steps, ws, device, rep=None):
    """The same steps with MX_OPT_PDL=2: layer l+1's CTAs start on the SMs
    layer l frees.  The layers of this workload are independent problems, so
    this is correct here, but a model whose layer l+1 reads layer l's output
    cannot overlap them: the headline value keeps the dependent order."""
    import torch

    from paper_2609_38386_gb300 import MX_OPT_PDL
    w.ctx.set_option(MX_OPT_PDL, 2)
    try:
        w.run_step()
        torch.cuda.synchronize(device)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            w.run_step()
        b.record()
        torch.cuda.synchronize(device)
        w.ctx.sync_status()
        ms = max_over_ranks(a.elapsed_time(b), ws, device)
    finally:
        w.ctx.set_option(MX_OPT_PDL, 1)
    return {"value": whole_job_value(w.tokens_per_step, steps, ws if rep is None else rep, ms), "unit": UNIT,
            "ms_per_step": ms / steps,
            "note": "MX_OPT_PDL=2: consecutive layers overlap (valid only for independent layers)"}


def graph_measure(w, device, stride=4):
    """Host enqueue cost of one iteration call with ordinary launches
    (mx_iteration) and replayed from a CUDA graph (mx_iteration_graph), on
    every stride-th iteration of the sweep, with the device times of both.
    The replayed launches read each layer's q/k/v up to the buffers'
    capacity, so this needs the lean layout (one buffer per layer, sized for
    the largest iteration), and one slot buffer that each call refreshes (the
    graph holds its pointer).  The first pass of each mode (the capture) is
    not counted."""
    import time

    import torch
    slots = torch.full((w.max_tok,), -1, dtype=torch.int32, device=device)
    idx = list(range(0, len(w.its), stride))
    gdescs = {}
    for i in idx:
        it = w.its[i]
        gdescs[i] = w.ctx.make_desc(decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
                                    prefill_seq_id=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t,
                                    page_table=w.page_table, slots=slots)
    out = {"iterations": len(idx), "layers": w.L}
    for mode in ("iteration", "graph"):
        enq, dev = [], []
        for rep in range(2):
            for i in idx:
                it = w.its[i]
                if mode == "graph":
                    slots[:it.n_tokens].copy_(w.slots[i])
                torch.cuda.synchronize(device)
                t0 = time.perf_counter()
                if mode == "graph":
                    w.ctx.iteration_graph(gdescs[i], w.layer_arrays[i], wait=False)
                else:
                    w.ctx.iteration(w.descs[i], w.layer_arrays[i], wait=False)
                t1 = time.perf_counter()
                torch.cuda.synchronize(device)
                us = (w.ctx.iteration_graph(gdescs[i], w.layer_arrays[i]) if mode == "graph"
                      else w.ctx.iteration(w.descs[i], w.layer_arrays[i]))
                if rep:
                    enq.append((t1 - t0) * 1e6)
                    dev.append(us)
        out[mode] = {"enqueue_us_mean": float(np.mean(enq)), "device_us_mean": float(np.mean(dev))}
    out["note"] = ("host time to enqueue one iteration call (planning, plan write, launches), and device time "
                   "per iteration; graph = mx_iteration_graph")
    return out


# Hidden and MLP widths of the Qwen3 models whose attention geometry each sweep
# uses (the models' published configurations).
MODEL_DIMS = {"qwen3-0.6b-attn-28L-chunk-sweep": (1024, 3072),
              "qwen3-8b-attn-36L-chunk-sweep": (4096, 12288),
              "qwen3-32b-attn-64L-chunk-sweep": (5120, 25600)}


def layer_measure(cfg, device, reps):
    """Whole decoder layers around the mixed attention (f3): for one
    iteration of each chunk size of the sweep (at the middle of the prompt)
    and the decode-only one, the device time of all n_layers layers (RMSNorm,
    QKV GEMM, QK norm + RoPE, mixed attention with the KV append, O GEMM +
    residual, RMSNorm, gate/up GEMM, SwiGLU, down GEMM + residual) against
    the attention alone on the same data.  One layer's random weights serve
    every layer (the KV pools are per layer); q/k/v are what the layer
    computes."""
    import torch

    from paper_2609_38386_gb300.layer import Qwen3Layer, positions_of
    d, f = MODEL_DIMS[cfg.name]
    w = Workload(cfg, device, lean=True)
    g = w.geom
    layer = Qwen3Layer(d, f, g.hq, g.hkv, seed=cfg.seed + 77, device=device)
    picks = {}
    for i, it in enumerate(w.its):
        if it.chunk_size not in picks or (it.chunk_size and it.chunk_start <= cfg.prompt_len // 2):
            picks[it.chunk_size] = i
    rows = []
    for p, i in sorted(picks.items()):
        it = w.its[i]
        n = it.n_tokens
        pos = torch.from_numpy(positions_of(it)).to(device)
        x = torch.empty((n, d), dtype=torch.int16, device=device)
        attns = []
        for l in range(w.L):
            q, k, v = w.inputs[i][l]
            kp, vp = w.pools[l]
            attns.append({"q": q, "k": k, "v": v, "k_pool": kp, "v_pool": vp, "out": w.outs[l]})
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        full = []
        for rep in range(reps + 1):
            x.copy_(torch.randn((n, d), device=device).to(torch.bfloat16).view(torch.int16))
            torch.cuda.synchronize(device)
            ev[0].record()
            for l in range(w.L):
                layer.forward(w.ctx, w.descs[i], x, pos, attns[l])
            ev[1].record()
            torch.cuda.synchronize(device)
            w.ctx.sync_status()
            if rep:
                full.append(ev[0].elapsed_time(ev[1]) * 1e3)
        att = [w.ctx.iteration(w.descs[i], w.layer_arrays[i]) for _ in range(reps + 1)][1:]
        fu, au = float(np.median(full)), float(np.median(att))
        rows.append({"p": it.p_t, "chunk_start": it.chunk_start, "tokens": n, "full_layers_us": fu,
                     "attention_us": au, "attention_share": au / fu, "tokens_per_s": n / fu * 1e6})
    w.close()
    return {"metric": "whole-layer iteration device us (all layers) and the attention share of L_t",
            "workload": f"{cfg.name.replace('-attn', '')}-full-layers", "d_model": d, "d_ffn": f,
            "layers": cfg.n_layers, "q_heads": g.hq, "kv_heads": g.hkv, "dtype": "bf16",
            "data": "synthetic (seeded random weights and activations)", "per_iteration": rows}


def several_chunks_measure(cfg, peaks, device, layers=28, reps=10):
    """Several prompts' chunks in one iteration (four 512-token chunks of
    four prompts at positions 1024/3072/5120/7168, plus the sweep's 32
    decodes) against the same decodes with one 2048-token chunk at 4096:
    device us per 28-layer iteration and the fraction of each iteration's
    roofline (the slower of its flops at the tensor peak and its bytes at
    the HBM peak)."""
    import numpy as np
    import torch

    import synth
    from paper_2609_38386_gb300 import Context
    from synth import device as sdev
    from synth import workload as wl
    g = cfg.geom
    it0 = [it for it in cfg.iterations() if it.chunk_size == 0][0]
    ctxs = [int(c) for c in it0.decode_ctx_lens]
    nd, npf, plen = len(ctxs), 4, 8192
    lay = wl.make_layout(g, [c + 1 for c in ctxs] + [plen] * npf, seed=cfg.seed + 991)
    ps = g.page_size
    pt_d = torch.from_numpy(lay.page_table).to(device)
    variants = {"four_512": [(nd + f, 1024 + 2048 * f, 512) for f in range(npf)],
                "one_2048": [(nd, 4096, 2048)]}
    n_tok = nd + 2048
    ctx = Context(num_q_heads=g.hq, num_kv_heads=g.hkv, num_pages=lay.num_pages, num_seqs=lay.num_seqs,
                  max_pages_per_seq=lay.max_pages, max_tokens=n_tok, max_decodes=nd, device=device.index or 0)
    bufs, keep = [], []
    for l in range(layers):
        t = {}
        for name, shape, kind in (("q", (n_tok, g.hq, g.head_dim), 0), ("k", (n_tok, g.hkv, g.head_dim), 1),
                                  ("v", (n_tok, g.hkv, g.head_dim), 2), ("kp", lay.pool_shape(), 3),
                                  ("vp", lay.pool_shape(), 4)):
            t[name] = torch.empty(shape, dtype=torch.int16, device=device)
            sdev.fill_(t[name], synth.stream_base(cfg.seed + 991, synth.stream_id(l, kind)))
        t["o"] = torch.empty((n_tok, g.hq, g.head_dim), dtype=torch.int16, device=device)
        keep.append(t)
        bufs.append(ctx.make_bufs(t["q"], t["k"], t["v"], t["kp"], t["vp"], t["o"]))
    arr = ctx.layer_array(bufs)
    out = {}
    for name, pfs in variants.items():
        slots = [lay.page_table[i, c // ps] * ps + c % ps for i, c in enumerate(ctxs)]
        B = F = 0
        for seq, cs, p in pfs:
            slots += [lay.page_table[seq, (cs + j) // ps] * ps + (cs + j) % ps for j in range(p)]
            b_, f_ = wl.algorithmic_work(g, wl.IterSpec(0, np.zeros(0, np.int32), np.zeros(0, np.int32),
                                                        seq, cs, p, p))
            B, F = B + b_, F + f_
        b_, f_ = wl.algorithmic_work(g, wl.IterSpec(0, it0.decode_seq_ids, it0.decode_ctx_lens, -1, 0, 0, 0))
        B, F = (B + b_) * layers, (F + f_) * layers
        sl_d = torch.from_numpy(np.asarray(slots, np.int32)).to(device)
        desc = ctx.make_desc(decode_seq_ids=list(range(nd)), decode_ctx_lens=ctxs, page_table=pt_d,
                             slots=sl_d, prefills=pfs)
        us = [ctx.iteration(desc, arr) for _ in range(reps + 3)][3:]
        ctx.sync_status()
        t_us = float(np.median(us))
        roof = max(F / (peaks["bf16_tflops_sustained"] * 1e12), B / (peaks["hbm_gbs"] * 1e9)) * 1e6
        out[name] = {"chunks": [[cs, p] for _, cs, p in pfs], "device_us_p50": t_us,
                     "roofline_us": roof, "roofline_frac": roof / t_us,
                     "tokens_per_s": (nd + sum(p for _, _, p in pfs)) / t_us * 1e6}
    ctx.close()
    del keep
    torch.cuda.empty_cache()
    return dict(out, note="32 decodes U[512,4096] + the chunks, 28 layers with distinct pools; "
                          "roofline from the measured peaks")


# ------------------------------------------------------------- CPU oracle
# Bounded samples of each sweep for the float64 CPU oracle: one layer call of
# one iteration (chunk size, chunk start), its first `decodes` decodes (None:
# all) and every `head_stride`-th query head (one per KV head at stride
# n_rep); the time is scaled by head_stride to all heads.
ORACLE_SAMPLES = {
    "qwen3-0.6b-attn-28L-chunk-sweep": {"light": (256, 4096, None, 1), "heavy": (2048, 6144, None, 1)},
    "qwen3-8b-attn-36L-chunk-sweep": {"light": (512, 4096, 32, 4), "heavy": (2048, 8192, 32, 4)},
    "qwen3-32b-attn-64L-chunk-sweep": {"light": (1024, 4096, 32, 8), "heavy": (4096, 8192, 32, 8)},
}


def oracle_sample(cfg, which="heavy"):
    """A bounded slice of the workload for the CPU oracle.  Returns (fn,
    tokens of the slice, description, time scale to all query heads)."""
    import oracle
    import synth
    from synth import workload as wl
    its = cfg.iterations()
    chunk, cs, n_dec, stride = ORACLE_SAMPLES.get(cfg.name, {}).get(which, (0, 0, None, 1))
    it = next((x for x in its if (x.chunk_size, x.chunk_start) == (chunk, cs)), its[-1])
    nd = it.n_decodes if n_dec is None else min(n_dec, it.n_decodes)
    it = wl.IterSpec(it.index, it.decode_seq_ids[:nd], it.decode_ctx_lens[:nd], it.prefill_seq,
                     it.chunk_start, it.p_t, it.chunk_size)
    lay = cfg.layout()
    g = cfg.geom
    q = np.ascontiguousarray(wl.host_tokens(cfg.seed, 0, synth.STREAM_Q, it, g.hq)[:, ::stride])
    k = wl.host_tokens(cfg.seed, 0, synth.STREAM_K, it, g.hkv)
    v = wl.host_tokens(cfg.seed, 0, synth.STREAM_V, it, g.hkv)
    # compact pool: the pages this slice reads or writes
    ps = g.page_size
    seqs = list(it.decode_seq_ids) + ([it.prefill_seq] if it.p_t else [])
    nkeys = list(it.decode_ctx_lens + 1) + ([it.chunk_start + it.p_t] if it.p_t else [])
    pages = np.unique(np.concatenate([lay.page_table[s, :-(-int(n) // ps)]
                                      for s, n in zip(seqs, nkeys)]))
    remap = np.full(lay.num_pages, -1, np.int64)
    remap[pages] = np.arange(len(pages))
    pe = g.hkv * ps * g.head_dim
    shp = (len(pages), g.hkv, ps, g.head_dim)
    kp0 = synth.values_pages(wl.pool_base(cfg.seed, 0, synth.STREAM_KPOOL), pages, pe).reshape(shp)
    vp0 = synth.values_pages(wl.pool_base(cfg.seed, 0, synth.STREAM_VPOOL), pages, pe).reshape(shp)
    pt = np.where(lay.page_table >= 0, remap[np.maximum(lay.page_table, 0)], -1).astype(np.int32)
    sl = it.slots(lay).astype(np.int64)
    sl = (remap[sl // ps] * ps + sl % ps).astype(np.int32)

    def fn():
        kp, vp = kp0.copy(), vp0.copy()
        oracle.mixed_attention(q=q, k=k, v=v, k_pool=kp, v_pool=vp, page_table=pt, slots=sl,
                               decode_seq_ids=it.decode_seq_ids,
                               decode_ctx_lens=it.decode_ctx_lens, prefill_seq=it.prefill_seq,
                               chunk_start=it.chunk_start, p_t=it.p_t)

    heads = (f"{g.hq // stride} of the {g.hq} query heads (one per KV head), time scaled x{stride} "
             "to all heads" if stride > 1 else f"all {g.hq} heads")
    desc = (f"one layer call of the p={it.p_t} iteration at chunk_start={it.chunk_start} "
            f"({nd} decodes + {it.p_t} chunk rows; {heads}); tokens/s scaled to the "
            f"{cfg.n_layers}-layer iteration")
    return fn, it.n_tokens, desc, stride


def cpu_baseline(cfg, which="heavy"):
    import oracle
    fn, ntok, desc, scale = oracle_sample(cfg, which)
    t0 = time.perf_counter()
    fn()
    dt = time.perf_counter() - t0
    return {"value": ntok / (dt * scale * cfg.n_layers), "unit": UNIT, "cores": oracle.max_threads(),
            "kind": "oracle", "sample": desc, "seconds": dt}


# ------------------------------------------------------------- DLFP trace
class TraceEngine:
    """Device state for an open-loop trace: per-layer pools with pages for
    every request's prompt and output, a page table with one row per request,
    q/k/v/out buffers sized for one iteration's token budget, and the
    completion-timed iteration call (`execute(plan) -> device us`)."""

    def __init__(self, requests, n_layers, hq, device, seed, budget, max_seqs):
        import torch

        import synth
        from paper_2609_38386_gb300 import Context
        from synth import device as sdev
        from synth import workload as wl
        self.geom = g = wl.Geometry(hq)
        caps = [r.prompt + r.output for r in requests]
        self.layout = lay = wl.make_layout(g, caps, seed=seed + 7)
        self.max_tok = budget + max_seqs
        self.ctx = Context(num_q_heads=hq, num_kv_heads=g.hkv, num_pages=lay.num_pages,
                           num_seqs=lay.num_seqs, max_pages_per_seq=lay.max_pages,
                           max_tokens=self.max_tok, max_decodes=max_seqs,
                           device=device.index or 0)
        self.page_table = torch.from_numpy(lay.page_table).to(device)
        self.slots_h = torch.empty(self.max_tok, dtype=torch.int32, pin_memory=True)
        self.slots_d = torch.empty(self.max_tok, dtype=torch.int32, device=device)
        self.keep = []
        bufs = []
        for l in range(n_layers):
            kp = torch.empty(lay.pool_shape(), dtype=torch.int16, device=device)
            vp = torch.empty_like(kp)
            sdev.fill_(kp, wl.pool_base(seed, l, synth.STREAM_KPOOL))
            sdev.fill_(vp, wl.pool_base(seed, l, synth.STREAM_VPOOL))
            q = torch.empty((self.max_tok, hq, g.head_dim), dtype=torch.int16, device=device)
            k = torch.empty((self.max_tok, g.hkv, g.head_dim), dtype=torch.int16, device=device)
            v = torch.empty_like(k)
            for t, kind in ((q, synth.STREAM_Q), (k, synth.STREAM_K), (v, synth.STREAM_V)):
                sdev.fill_(t, synth.stream_base(seed, synth.stream_id(l, kind, 7)))
            out = torch.empty_like(q)
            self.keep.append((kp, vp, q, k, v, out))
            bufs.append(self.ctx.make_bufs(q, k, v, kp, vp, out))
        self.layers = self.ctx.layer_array(bufs)
        torch.cuda.synchronize(device)
        self.iterations = 0

    def execute(self, plan):
        import numpy as np
        lay = self.layout
        parts = [lay.slot(rid, ctx)[None] for rid, ctx in zip(plan.decode_ids, plan.decode_ctx)]
        if plan.p_t:
            parts.append(lay.slot(plan.prefill_id,
                                  np.arange(plan.chunk_start, plan.chunk_start + plan.p_t)))
        n = len(plan.decode_ids) + plan.p_t
        if n:
            self.slots_h[:n].copy_(__import__("torch").from_numpy(np.concatenate(parts)))
            self.slots_d[:n].copy_(self.slots_h[:n], non_blocking=True)
        desc = self.ctx.make_desc(decode_seq_ids=plan.decode_ids, decode_ctx_lens=plan.decode_ctx,
                                  prefill_seq_id=plan.prefill_id, chunk_start=plan.chunk_start,
                                  p_t=plan.p_t, page_table=self.page_table, slots=self.slots_d)
        self.iterations += 1
        return self.ctx.iteration(desc, self.layers)


def trace_measure(device, seeds=(801, 802, 803), n_layers=28, hq=16, budget=8192,
                  max_seqs=64, fixed_caps=(2048, 3072, 4096), loads=(20.0, 5.0)):
    """Config 5: the completion-timed DLFP loop against fixed chunk caps on
    seeded open-loop traces (§3.1 Eq. 2 with L_t = device-completion time).
    `loads` are mean inter-arrival times in units of t_ref (20 is the
    reference load; smaller is heavier)."""
    import numpy as np
    import torch

    from paper_2609_38386_gb300 import dlfp
    # t_ref: 16 decodes at context 1024 beside a 2048-token chunk at position 0
    cal_reqs = [dlfp.Request(i, 0.0, 1025, 2) for i in range(16)] + [dlfp.Request(16, 0.0, 2048, 1)]
    eng = TraceEngine(cal_reqs, n_layers, hq, device, 0, budget, max_seqs)
    cal = dlfp.IterationPlan(list(range(16)), [1024] * 16, 16, 0, 2048, None)
    for _ in range(3):
        eng.execute(cal)
    t_ref = float(np.median([eng.execute(cal) for _ in range(7)]))
    del eng
    torch.cuda.empty_cache()
    result = {"t_ref_us": t_ref, "target_us": t_ref, "fixed_caps": list(fixed_caps), "loads": {}}
    policies = [f"fixed{c}" for c in fixed_caps] + ["dlfp"]
    for load in loads:
        per_load = {"mean_interarrival_us": load * t_ref, "seeds": {}}
        red = {f"fixed{c}": [] for c in fixed_caps}
        for seed in seeds:
            spec = dlfp.TraceSpec(mean_interarrival=load * t_ref, seed=seed)
            eng = TraceEngine(spec.requests(), n_layers, hq, device, seed, budget, max_seqs)
            per = {}
            for name in policies:
                ctl = (dlfp.DLFPController(t_ref) if name == "dlfp"
                       else dlfp.FixedCap(int(name[len("fixed"):])))
                sch = dlfp.Scheduler(spec.requests(), ctl, max_seqs=max_seqs, budget=budget)
                t0 = time.perf_counter()
                per[name] = sch.run(eng.execute)
                per[name]["wall_s"] = time.perf_counter() - t0
            for c in fixed_caps:
                red[f"fixed{c}"].append(1 - per["dlfp"]["itl_p99"] / per[f"fixed{c}"]["itl_p99"])
            per_load["seeds"][str(seed)] = per
            del eng
            torch.cuda.empty_cache()
        per_load["mean_itl_p99_reduction_vs"] = {k: float(np.mean(v)) for k, v in red.items()}
        result["loads"][f"{load:g}"] = per_load
    return result


# ---------------------------------------------------------------- timing
def time_sweep(w, steps, warmup, ws, device, barrier, sampler=None):
    """W untimed steps, then K timed steps bracketed by a barrier and a
    synchronise on both sides; CUDA events on the launching stream around
    the whole region and around every iteration.  Returns (max-over-ranks
    total ms, per-iteration device us [steps][iterations], clocks)."""
    import torch
    for _ in range(max(warmup, 0)):
        w.run_step()
    w.ctx.sync_status()
    torch.cuda.synchronize(device)
    n_it = len(w.its)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_it + 1)] for _ in range(steps)]
    barrier()
    torch.cuda.synchronize(device)
    if sampler is not None:
        sampler.start()
        time.sleep(0.25)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record()
    for s_ in range(steps):
        w.run_step(evs[s_])
    t_end.record()
    torch.cuda.synchronize(device)
    clocks = sampler.stop() if sampler is not None else None
    barrier()
    w.ctx.sync_status()
    total_ms = max_over_ranks(t_start.elapsed_time(t_end), ws, device)
    it_us = np.array([[evs[s_][i].elapsed_time(evs[s_][i + 1]) * 1e3 for i in range(n_it)]
                      for s_ in range(steps)])
    return total_ms, it_us, clocks


def summarize(w, it_us, peaks, config_name):
    """Per chunk size: device us P50/P99 per iteration, tokens/s, the
    fraction of the iterations' roofline (the slower of their flops at the
    sustained tensor peak and their bytes at the HBM peak), P99 against the
    decode-only iteration; and the roofline object of the whole sweep."""
    n_it = len(w.its)
    L = w.L
    hbm = peaks["hbm_gbs"] * 1e9
    tfl = peaks["bf16_tflops_sustained"] * 1e12
    B = np.array([L * b for b, _ in w.work], dtype=np.float64)
    F = np.array([L * f for _, f in w.work], dtype=np.float64)
    t_it = it_us.mean(axis=0) * 1e-6                         # seconds per iteration
    per_chunk = {}
    p0_p99 = None
    for p in sorted(set(it.chunk_size for it in w.its)):
        idx = [i for i, it in enumerate(w.its) if it.chunk_size == p]
        samples = it_us[:, idx].ravel()
        toks = sum(w.its[i].n_tokens for i in idx)
        t_sum = t_it[idx].sum()
        roof = sum(max(F[i] / tfl, B[i] / hbm) for i in idx)
        p99 = float(np.percentile(samples, 99))
        if p == 0:
            p0_p99 = p99
        # beside the measured peaks: the nominal 8 TB/s and 1706.7 TFLOP/s
        # sustained, and the bound with no HBM/tensor overlap at all
        roof_spec = sum(max(F[i] / SPEC_TFLOPS, B[i] / SPEC_HBM) for i in idx)
        no_overlap = sum(F[i] / tfl + B[i] / hbm for i in idx)
        per_chunk[str(p)] = {
            "iterations": len(idx), "samples": int(samples.size),
            "device_us_p50": float(np.percentile(samples, 50)), "device_us_p99": p99,
            "tokens_per_s": toks / t_sum,
            "roofline_us_per_iter": roof / len(idx) * 1e6,
            "roofline_frac": roof / t_sum,
            "roofline_frac_spec": roof_spec / t_sum,
            "no_overlap_us_per_iter": no_overlap / len(idx) * 1e6,
            "no_overlap_frac": no_overlap / t_sum,
            "bound": "tensor" if sum(F[idx]) / tfl > sum(B[idx]) / hbm else "hbm",
            "hbm_gbs": float(B[idx].sum() / t_sum / 1e9),
            "tflops": float(F[idx].sum() / t_sum / 1e12)}
    if p0_p99:
        for v in per_chunk.values():
            v["p99_vs_decode_only"] = v["device_us_p99"] / p0_p99
    t_total = t_it.sum()
    bound = "tensor" if F.sum() / tfl > B.sum() / hbm else "hbm"
    if bound == "hbm":
        achieved, peak, unit = B.sum() / t_total / 1e9, peaks["hbm_gbs"], "GB/s"
        peak_kind = "measured HBM copy" if peaks["source"] == "measured" else "fallback HBM"
    else:
        achieved, peak, unit = F.sum() / t_total / 1e12, peaks["bf16_tflops_sustained"], "TFLOP/s"
        peak_kind = ("measured sustained bf16 GEMM" if peaks["source"] == "measured"
                     else "fallback sustained bf16")
    roofline = {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                "frac": achieved / peak, "traffic": committed_traffic(config_name),
                "algorithmic_bytes_per_launch": float(B.sum() / (L * n_it)),
                "algorithmic_flops_per_launch": float(F.sum() / (L * n_it)),
                "avg_launch_us": float(t_total / (L * n_it) * 1e6),
                "max_bound_frac": float(sum(max(F[i] / tfl, B[i] / hbm) for i in range(n_it))
                                        / t_total),
                "peak_source": peaks["source"], "peak_kind": peak_kind,
                "kernel": "mixed_layer_kernel"}
    return per_chunk, roofline


def side_config(name, steps, warmup, peaks, device, barrier):
    """Another sweep in the same run, reported beside the headline."""
    import torch
    from synth import workload as wl
    cfg = wl.CONFIGS[name]
    w = Workload(cfg, device, lean=name in LEAN_CONFIGS)
    total_ms, it_us, _ = time_sweep(w, steps, warmup, 1, device, barrier)
    per_chunk, roofline = summarize(w, it_us, peaks, name)
    out = {"value": whole_job_value(w.tokens_per_step, steps, 1, total_ms), "unit": UNIT,
           "steps": steps, "warmup": warmup, "ms_per_step": total_ms / steps,
           "layers": cfg.n_layers, "q_heads": cfg.hq, "decodes": cfg.n_decodes,
           "prompt_len": cfg.prompt_len, "iterations_per_step": len(w.its),
           "roofline": roofline, "per_chunk": per_chunk}
    w.close()
    del w
    torch.cuda.empty_cache()
    return out


# ------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--profile", action="store_true",
                    help="small case for ncu: 2 layers, iterations of --profile-chunk only")
    ap.add_argument("--profile-chunk", type=int, default=2048)
    ap.add_argument("--layers", type=int, default=0,
                    help="run only the first N layers of every iteration (for launch-list captures: "
                         "each launch does the same work as in the full sweep, on its own layer's pool)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-side", action="store_true", help="skip the sweeps reported beside the headline")
    ap.add_argument("--lean", action="store_true",
                    help="one q/k/v buffer per layer reused by all iterations (large sweeps)")
    ap.add_argument("--shard", default="none", choices=["none", "kv"],
                    help="kv (N > 1): each rank runs 1/N of the KV heads (and their query groups) of the "
                         "same tokens: tensor parallelism of attention, strong scaling, no collective "
                         "inside attention; default: N independent replicas (weak scaling)")
    ap.add_argument("--workload", default="sweep", choices=["sweep", "trace", "layer"],
                    help="trace: the completion-timed DLFP loop vs a fixed chunk cap; layer: whole "
                         "Qwen3 layers (random weights) around the attention on iterations of --config")
    args = ap.parse_args()

    ws, rank, local = dist_setup()
    from synth import workload as wl
    cfg = wl.CONFIGS[args.config]
    sharded = args.shard == "kv" and ws > 1
    if sharded:
        import dataclasses
        if cfg.hkv % ws:
            raise SystemExit(f"--shard kv needs the {cfg.hkv} KV heads to divide among {ws} ranks")
        cfg = dataclasses.replace(cfg, hq=cfg.hq // ws, hkv=cfg.hkv // ws)
    # every rank processes its own tokens (replicas) or the same tokens (KV-head shards)
    rep = 1 if sharded else ws
    lean = args.lean or args.config in LEAN_CONFIGS
    config = {"workload": cfg.name, "q_heads": cfg.hq * (ws if sharded else 1),
              "kv_heads": cfg.hkv * (ws if sharded else 1), "head_dim": 128,
              "page_size": 16, "layers": cfg.n_layers, "decodes": cfg.n_decodes,
              "decode_ctx": f"{cfg.ctx_dist}[{cfg.ctx_lo},{cfg.ctx_hi}]",
              "prompt_len": cfg.prompt_len, "chunk_sizes": list(cfg.chunk_sizes),
              "iterations_per_step": len(cfg.iterations()),
              "l2": f"inputs larger than L2: each iteration reads {cfg.n_layers} distinct "
                    "per-layer KV pools of several hundred MB or more",
              "parallelism": f"kv-heads{ws}" if sharded else f"replicas{ws}"}

    if args.impl == "reference":
        if rank != 0:
            return
        import oracle
        fn, ntok, desc, scale = oracle_sample(cfg, "light")
        for _ in range(args.warmup):
            fn()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            fn()
        dt = time.perf_counter() - t0
        val = ntok * args.steps / (dt * scale * cfg.n_layers)
        line = {"impl": "reference", "metric": METRIC, "value": val, "unit": UNIT,
                "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": dt * 1e3 / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": config,
                "cpu_baseline": {"value": val, "unit": UNIT, "cores": oracle.max_threads(),
                                 "kind": "oracle", "sample": desc},
                "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import torch
    if args.workload == "trace":
        if rank == 0:
            device = torch.device("cuda", local)
            torch.cuda.set_device(device)
            res = trace_measure(device)
            print(json.dumps({"metric": "open-loop trace: per-iteration device us P50/P99 and "
                              "ITL/TTFT, completion-timed DLFP vs fixed chunk caps",
                              "workload": "qwen3-0.6b-attn-28L-poisson-trace", **res}))
        return
    if args.workload == "layer":
        if rank == 0:
            device = torch.device("cuda", local)
            torch.cuda.set_device(device)
            print(json.dumps(layer_measure(cfg, device, max(1, args.steps))))
        return
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    peaks = load_peaks()

    layers = 2 if args.profile else (args.layers or None)
    w = Workload(cfg, device, seed_offset=replica_seed_offset(rank), layers=layers, lean=lean)
    if lean:
        config["inputs"] = "one q/k/v buffer per layer, reused by every iteration"
    if args.profile:
        keep = [i for i, it in enumerate(w.its) if it.chunk_size == args.profile_chunk][-2:]
        w.its = [w.its[i] for i in keep]
        w.descs = [w.descs[i] for i in keep]
        w.layer_arrays = [w.layer_arrays[i] for i in keep]
        w.work = [w.work[i] for i in keep]
        w.inputs = [w.inputs[i] for i in keep]
        w.tokens_per_step = sum(it.n_tokens for it in w.its)
        config["workload"] += f"-profile-{w.L}L-p{args.profile_chunk}"
    elif args.layers:
        config["workload"] += f"-first-{w.L}L"
        config["layers"] = w.L

    def barrier():
        if ws > 1:
            torch.distributed.barrier()

    gpu_id = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
    total_ms, it_us, clocks = time_sweep(w, args.steps, args.warmup, ws, device, barrier,
                                         ClockSampler(gpu_id))
    per_chunk, roofline = summarize(w, it_us, peaks, args.config if not args.profile else None)
    n_it = len(w.its)
    value = whole_job_value(w.tokens_per_step, args.steps, rep, total_ms)
    plan = w.ctx.last_plan()
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
            "higher_is_better": True, "scaling": "strong" if sharded else "weak", "vs_baseline": None,
            "dtype": "bf16",
            "data": "synthetic (seeded N(0,1) bf16, random page permutation)",
            "config": config, "roofline": roofline, "per_chunk": per_chunk,
            # per iteration: one plan-upload kernel and one mixed_layer_kernel per layer
            "gpu_launches": (w.L + 1) * n_it * args.steps, "clocks": clocks,
            "plan_last": plan}
    if not args.no_e2e and not args.profile:
        line["e2e"] = e2e_measure(w, max(1, min(args.steps, 3)), device)
    if not args.profile:
        line["independent_layers"] = independent_layers_measure(w, max(1, min(args.steps, 3)), ws, device, rep)
        if args.config in LEAN_CONFIGS or args.lean:
            line["graph"] = graph_measure(w, device)
    if rank == 0 and ws == 1 and not args.no_cpu and not args.profile:
        line["cpu_baseline"] = cpu_baseline(cfg)
    w.close()
    del w
    torch.cuda.empty_cache()
    if not args.profile and not args.no_side and ws == 1:
        side = {}
        for name in SIDE_CONFIGS:
            if name != args.config:
                side[name] = side_config(name, max(1, min(args.steps, 5)), 2, peaks, device, barrier)
        line["other_configs"] = side
        if "qwen3-0.6b-attn-28L-chunk-sweep" in wl.CONFIGS:
            line["several_chunks"] = several_chunks_measure(wl.CONFIGS["qwen3-0.6b-attn-28L-chunk-sweep"],
                                                            peaks, device)
    if rank == 0:
        print(json.dumps(line))
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
