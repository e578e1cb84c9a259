"""Benchmark of the packed-cache attention step on GB300.

One step is one pass of the whole path over one batch of the default workload,
the Llama-3.1-8B-shaped attention stack (32 layers, batch 16, hidden 4096, 32
query / 8 KV heads, head_dim 128, RoPE base 500000, KIVI K2V2 cache with groups
of 32 and a 128-token full-precision residual, rank-16 LoRA on Q, K and V):
reset the caches, prefill 8192 tokens per sequence (LoRA Q/K/V projection with
RoPE, quantize-and-pack append, causal prefill attention, per layer), then 64
decode steps (projection, append, split-K decode attention through
kvq_decode_step; one captured CUDA graph per decode step).  `value` is tokens
processed per second (batch x (prefill + decode) tokens per step); the decode
phase alone, the packed-cache decode attention against HBM, pack bandwidth and
projection TFLOP/s are reported beside it.  --workload selects another shape
(the TinyLlama-shaped affine/symmetric stacks, the 12B-class KVarN stack, the
single fp32 layer).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl kvq|reference]

--impl reference times the CPU oracle on the host cores over a bounded sample
of the same workload.  Under torchrun each rank runs an independent replica
(the path has no exchange step); rank 0 prints the JSON line.
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

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2609_04263_gb300 import synth  # noqa: E402

METRIC = ("packed-KV decode attention tokens/s and % HBM roofline; pack GB/s; "
          "QKV TFLOP/s")
WORKLOAD = "llama8b_kivi"
PEAKS_PATH = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


TRAFFIC_PATH = os.path.join(ROOT, "profiles", "roofline_traffic.json")


def measured_traffic(workload, kernel, variant=""):
    """DRAM bytes per launch of `kernel` on `workload` from the committed ncu
    record (keyed "workload/kernel[/variant]"), or None when there is none or
    the kernel's sources changed since it was taken."""
    import hashlib
    key = f"{workload}/{kernel}" + (f"/{variant}" if variant else "")
    try:
        with open(TRAFFIC_PATH) as f:
            rec = json.load(f)[key]
        h = hashlib.sha256()
        for name in rec["sources"]:
            with open(os.path.join(ROOT, name), "rb") as f:
                h.update(f.read())
    except (OSError, KeyError, ValueError):
        return None
    return rec["dram_bytes_per_launch"] if h.hexdigest() == rec["sources_sha256"] else None


def load_peaks():
    try:
        with open(PEAKS_PATH) as f:
            return json.load(f), "measured"
    except OSError:
        return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------------------
# algorithmic work per launch (numerators of the roofline)
# ---------------------------------------------------------------------------
def code_bytes_per_token(wl):
    """Packed bytes one token adds per KV head (codes + fp16 metadata)."""
    D, G = wl.head_dim, wl.group_size
    meta = 2 if wl.fmt == synth.FMT_SYMMETRIC else 4
    return D * (wl.key_bits + wl.value_bits) // 8 + 2 * (D // G) * meta


def proj_flops(wl, M):
    D = wl.head_dim
    N = wl.n_out
    douts = (wl.n_q_heads * D, wl.n_kv_heads * D, wl.n_kv_heads * D)
    r = wl.rank
    return 2 * M * wl.d_in * N + 2 * M * wl.d_in * 3 * r + 2 * M * r * sum(douts)


def proj_bytes(wl, M):
    """HBM bytes of a projection launch: weights, LoRA factors, x, outputs."""
    D, r = wl.head_dim, wl.rank
    w = wl.n_out * wl.d_in
    lora = 3 * r * wl.d_in + r * wl.n_out
    return 2 * (w + lora + M * wl.d_in + M * wl.n_out)


def coded_bytes_per_token(wl):
    """Packed bytes per coded token and KV head, with KVarN's fp16 row scale and
    its share of the per-block fp16 column scales (keys and values)."""
    extra = 2 * (2 + 2 * wl.head_dim // wl.group_size) if wl.fmt == synth.FMT_KVARN else 0
    return code_bytes_per_token(wl) + extra


def cache_read_bytes(wl, T):
    """HBM bytes a decode attention reads from one (sequence, KV head) holding
    T tokens: coded tokens plus the full-precision windows (KIVI residual,
    KVarN sinks and staged tokens) in the activation dtype."""
    G = wl.group_size
    full = 2 * wl.head_dim * (2 if wl.dtype == "bf16" else 4)
    if wl.fmt == synth.FMT_FLOAT:
        return T * full
    coded = coded_bytes_per_token(wl)
    if wl.fmt == synth.FMT_KIVI:
        tq = G * (max(T - wl.residual_tokens, 0) // G)
        return tq * coded + (T - tq) * full
    if wl.fmt == synth.FMT_KVARN:
        s = min(T, wl.sink_tokens)
        tq = G * ((T - s) // G)
        return tq * coded + (T - tq) * full
    return T * coded


def pack_bytes(wl, L):
    B, H, D = wl.batch, wl.n_kv_heads, wl.head_dim
    return B * H * L * (2 * D * 2 + coded_bytes_per_token(wl))


def decode_attn_bytes(wl, T):
    B, H, Hq, D = wl.batch, wl.n_kv_heads, wl.n_q_heads, wl.head_dim
    return B * H * cache_read_bytes(wl, T) + 2 * B * Hq * D * 2


def decode_step_bytes(wl, T):
    """HBM bytes of one fused decode step of one layer: the projection's
    weights, factors, input and q/k/v outputs, the new token's packed codes,
    the cache read by attention over T tokens and its output."""
    B, H = wl.batch, wl.n_kv_heads
    return proj_bytes(wl, B) + B * H * code_bytes_per_token(wl) + decode_attn_bytes(wl, T)


def prefill_attn_flops(wl, L, T):
    """Causal: query l (position T - L + l) sees T - L + l + 1 keys; QK^T and
    PV each 2 D flops per visible key."""
    B, Hq, D = wl.batch, wl.n_q_heads, wl.head_dim
    visible = L * (T - L) + L * (L + 1) // 2
    return 4 * B * Hq * D * visible


# ---------------------------------------------------------------------------
# the GPU path
# ---------------------------------------------------------------------------
class Runner:
    def __init__(self, wl: synth.Workload, device: str):
        from paper_2609_04263_gb300 import api
        self.api, self.wl, self.dev = api, wl, device
        dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        self.dt = dt
        B, P, Dn, D = wl.batch, wl.prefill, wl.decode, wl.head_dim
        self.layers = []
        for l in range(wl.layers):
            w, lora = synth.layer_weights(wl, l)
            self.layers.append((
                torch.from_numpy(w).to(dt).to(device),
                {p: tuple(torch.from_numpy(t).to(dt).to(device) for t in lora[p]) for p in "qkv"},
            ))
        desc = api.make_desc(wl.fmt, wl.key_bits, wl.value_bits, wl.group_size, B,
                             wl.n_kv_heads, wl.n_q_heads, D, wl.max_tokens, dt,
                             residual_tokens=wl.residual_tokens, sink_tokens=wl.sink_tokens,
                             norm_iters=wl.norm_iters)
        self.caches = [api.Cache(desc, device=device) for _ in range(wl.layers)]
        self.cache_bytes = self.caches[0].nbytes
        x_pre = synth.hidden_states((B, P, wl.d_in), wl.hidden, wl.outlier_frac, seed=0)
        x_dec = synth.hidden_states((B, Dn, wl.d_in), wl.hidden, wl.outlier_frac, seed=0,
                                    stream=1)
        self.x_pre_host = torch.from_numpy(x_pre).to(dt).pin_memory()
        self.x_dec_host = torch.from_numpy(
            np.ascontiguousarray(x_dec.transpose(1, 0, 2)[:, :, None, :])).to(dt).pin_memory()
        self.x_pre = self.x_pre_host.to(device)
        self.x_dec = self.x_dec_host.to(device)         # [Dn, B, 1, d_in]
        Hq, Hkv = wl.n_q_heads, wl.n_kv_heads
        e = lambda *s: torch.empty(*s, dtype=dt, device=device)
        self.pre = (e(B, Hq, P, D), e(B, Hkv, P, D), e(B, Hkv, P, D))
        self.o_pre = e(B, Hq, P, D)
        self.xs = e(B, 1, wl.d_in)
        self.dec = (e(B, Hq, 1, D), e(B, Hkv, 1, D), e(B, Hkv, 1, D))
        self.o_dec = e(B, Hq, 1, D)
        self.graph = None
        self.events = None
        self.eager = False
        # decode steps through kvq_decode_step (one fused kernel per layer
        # where the cache format allows) unless separate calls are asked for
        self.separate = False
        self.fused = self.caches[0].decode_step_fused(wl.d_in, self.layers[0][1])
        # prefill: projection fused with the append where the cache format allows
        self.fused_append = self.caches[0].project_append_supported(P, wl.d_in, self.layers[0][1])

    # one layer's calls ----------------------------------------------------
    def _project(self, l, x, out):
        w, lora = self.layers[l]
        wl = self.wl
        return self.api.project_lora(x, w, lora, wl.alpha_over_r, wl.n_q_heads, wl.n_kv_heads,
                                     wl.head_dim, rope_base=wl.rope_base, out=out,
                                     pos_cache=self.caches[l])

    def reset(self):
        for c in self.caches:
            c.reset()

    def prefill(self, timer=None):
        for l, c in enumerate(self.caches):
            if self.fused_append:
                # one kernel projects and codes the new keys and values into the cache
                w, lora = self.layers[l]
                if timer:
                    timer("project", 0)
                q = c.project_append(self.x_pre, w, lora, self.wl.alpha_over_r, self.wl.rope_base,
                                     q=self.pre[0])
                if timer:
                    timer("project", 1)
                    timer("attend_prefill", 0)
                c.attend_prefill(q, out=self.o_pre)
                if timer:
                    timer("attend_prefill", 1)
                continue
            if timer:
                timer("project", 0)
            q, k, v = self._project(l, self.x_pre, self.pre)
            if timer:
                timer("project", 1)
                timer("append", 0)
            c.append(k, v)
            if timer:
                timer("append", 1)
                timer("attend_prefill", 0)
            c.attend_prefill(q, out=self.o_pre)
            if timer:
                timer("attend_prefill", 1)

    def decode_step_eager(self, timer=None):
        if not self.separate:
            wl = self.wl
            for l, c in enumerate(self.caches):
                w, lora = self.layers[l]
                if timer:
                    timer("decode_step", 0)
                c.decode_step(self.xs, w, lora, wl.alpha_over_r, wl.rope_base, qkv=self.dec,
                              out=self.o_dec)
                if timer:
                    timer("decode_step", 1)
            return
        for l, c in enumerate(self.caches):
            if timer:
                timer("project_decode", 0)
            q, k, v = self._project(l, self.xs, self.dec)
            if timer:
                timer("project_decode", 1)
                timer("append_decode", 0)
            c.append(k, v)
            if timer:
                timer("append_decode", 1)
                timer("attend_decode", 0)
            c.attend_decode(q, out=self.o_dec)
            if timer:
                timer("attend_decode", 1)

    def decode_step_layers(self):
        wl = self.wl
        for l, c in enumerate(self.caches):
            w, lora = self.layers[l]
            c.decode_step(self.xs, w, lora, wl.alpha_over_r, wl.rope_base, qkv=self.dec,
                          out=self.o_dec)

    # the three decode call classes, each over all layers (for timing)
    def decode_project_layers(self):
        for l in range(len(self.caches)):
            self._project(l, self.xs, self.dec)

    def decode_append_layers(self):
        for c in self.caches:
            c.append(self.dec[1], self.dec[2])

    def decode_attend_layers(self):
        for c in self.caches:
            c.attend_decode(self.dec[0], out=self.o_dec)

    def capture(self):
        """Capture one decode step (all layers) in a CUDA graph."""
        self.reset()
        self.prefill()                       # the caches' device state is initialised
        torch.cuda.synchronize()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            self.decode_step_eager()
        torch.cuda.synchronize()
        self.graph = g

    def decode(self):
        for s in range(self.wl.decode):
            self.xs.copy_(self.x_dec[s])
            if self.eager:
                self.decode_step_eager()
            else:
                self.graph.replay()

    def job(self, phase_events=None):
        self.reset()
        if phase_events:
            phase_events[0].record()
        self.prefill()
        if phase_events:
            phase_events[1].record()
        self.decode()
        if phase_events:
            phase_events[2].record()

    def job_e2e(self, x_pre_host, x_dec_host, o_host, od_host, copy_stream):
        """One job through the public API with host buffers: the step's inputs
        go up from pinned host memory and its outputs come back, inside the
        step.  x_pre (read by every layer's projection) goes up first on the
        compute stream; x_dec goes up on `copy_stream` during the prefill, and
        the prefill output comes back on it while the decode steps run (they
        do not touch it); the step ends when both streams are done."""
        cur = torch.cuda.current_stream()
        copy_stream.wait_stream(cur)
        self.x_pre.copy_(x_pre_host, non_blocking=True)
        with torch.cuda.stream(copy_stream):
            self.x_dec.copy_(x_dec_host, non_blocking=True)
        x_dec_up = torch.cuda.Event()
        x_dec_up.record(copy_stream)
        self.reset()
        self.prefill()
        prefilled = torch.cuda.Event()
        prefilled.record(cur)
        copy_stream.wait_event(prefilled)
        with torch.cuda.stream(copy_stream):
            o_host.copy_(self.o_pre, non_blocking=True)
        cur.wait_event(x_dec_up)
        self.decode()
        od_host.copy_(self.o_dec, non_blocking=True)
        cur.wait_stream(copy_stream)

    def decode_path(self):
        if self.separate:
            return "three calls per layer (project, append, attend)"
        return ("kvq_decode_step: one fused kernel per layer" if self.fused else
                "kvq_decode_step: three kernels per layer")

    def traffic_variant(self):
        """Which decode-step implementation the per-kernel "decode_step" times."""
        return "separate" if self.separate else ("fused" if self.fused else "three_kernels")

    def kvarn_streamed(self):
        """Whether KVarN decode attention at the prefill length takes the
        tensor-core kernel over the coded tokens (the library's size rule)."""
        wl = self.wl
        if wl.fmt != synth.FMT_KVARN or wl.dtype != "bf16" or (wl.key_bits, wl.value_bits) != (4, 2):
            return False
        if (wl.head_dim, wl.group_size) not in ((256, 64), (64, 32)):
            return False
        bh = wl.batch * wl.n_kv_heads
        ctas = min(torch.cuda.get_device_properties(0).multi_processor_count, 15 * bh)
        coded = max(wl.prefill - wl.sink_tokens, 0) // wl.group_size * wl.group_size
        return bh * (coded // 32) >= 16 * ctas

    def launches_per_step(self):
        """Kernels the library launches in one whole-job step."""
        wl = self.wl
        append = {synth.FMT_FLOAT: 1, synth.FMT_AFFINE: 1, synth.FMT_SYMMETRIC: 1,
                  synth.FMT_KIVI: 3, synth.FMT_KVARN: 2}[wl.fmt]
        # decode attention merges its splits in its last CTA on the
        # tensor-core path (bf16, affine/symmetric/KIVI), else in a second kernel
        attend = 1 if (wl.dtype == "bf16" and wl.fmt in (synth.FMT_AFFINE, synth.FMT_SYMMETRIC,
                                                         synth.FMT_KIVI)
                       and wl.head_dim in (64, 128)) else 2
        if self.kvarn_streamed():
            attend = 3          # coded tokens, sinks and staged tokens, combine
        prefill = wl.layers * (2 if self.fused_append else 1 + append + 1)
        per_layer = 1 if (self.fused and not self.separate) else 1 + append + attend
        return prefill + wl.decode * wl.layers * per_layer


class EventTimer:
    """Per-call-class CUDA events on the current stream."""

    def __init__(self):
        self.open = {}
        self.pairs = {}

    def __call__(self, name, edge):
        ev = torch.cuda.Event(enable_timing=True)
        ev.record()
        if edge == 0:
            self.open[name] = ev
        else:
            self.pairs.setdefault(name, []).append((self.open.pop(name), ev))

    def mean_ms(self):
        torch.cuda.synchronize()
        return {k: statistics.mean(a.elapsed_time(b) for a, b in v) for k, v in self.pairs.items()}

    def total_ms(self):
        torch.cuda.synchronize()
        return {k: sum(a.elapsed_time(b) for a, b in v) for k, v in self.pairs.items()}


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index, self.proc, self.path = index, None, None

    def start(self):
        import tempfile
        out_dir = tempfile.mkdtemp(prefix="kvq_clocks_")
        self.path = os.path.join(out_dir, f"clocks_rank{self.index}.csv")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait(timeout=10)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        import shutil
        shutil.rmtree(os.path.dirname(self.path), ignore_errors=True)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "samples": len(sm), "reasons": sorted(reasons)}


def l2_flush(buf):
    """Write the first half (256 MiB, twice L2), then read the second: the
    read evicts the written lines, so their write-back happens here and not
    inside the next timed kernel, which starts with a cold, clean L2."""
    half = buf.numel() // 2
    buf[:half].fill_(1)
    buf[half:].view(torch.float32).sum()      # a plain reduction: no widened copy


def graph_time_ms(fn, reps):
    """Mean device time of one call of `fn` (a sequence of launches), from a
    captured graph replayed `reps` times between CUDA events (two untimed
    replays first)."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        fn()
    torch.cuda.synchronize()
    for _ in range(2):
        g.replay()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        g.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def cold_graph_time_ms(fn, reps, flush):
    """Mean device time of one call of `fn` replayed from a captured graph,
    with L2 flushed before each timed replay (outside the events)."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        fn()
    torch.cuda.synchronize()
    g.replay()
    ms = []
    for _ in range(reps):
        l2_flush(flush)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        g.replay()
        b.record()
        torch.cuda.synchronize()
        ms.append(a.elapsed_time(b))
    return statistics.mean(ms)


def nf4_projection_rates(run, peaks, flush):
    """The projection of layer 0 over an NF4 base (kvq_project_lora_nf4) at the
    workload's prefill rows (tensor bound) and decode rows (HBM bound: codes,
    absmax, LoRA factors, x and outputs), beside the bf16-base rows above.
    None when the head shapes are outside the NF4 kernel's range."""
    wl = run.wl
    D = wl.head_dim
    if D not in (64, 128) or (wl.n_q_heads * D) % 128 or (wl.n_kv_heads * D) % 128:
        return None
    codes, absmax = synth.nf4_base(wl, 0)
    tc = torch.from_numpy(codes).to(run.dev)
    ta = torch.from_numpy(absmax).to(run.dev)
    lora = run.layers[0][1]
    args = (wl.alpha_over_r, wl.n_q_heads, wl.n_kv_heads, D)

    def pre():
        run.api.project_lora_nf4(run.x_pre, tc, ta, lora, *args, rope_base=wl.rope_base,
                                 out=run.pre)

    def dec():
        run.api.project_lora_nf4(run.xs, tc, ta, lora, *args, pos0=wl.prefill,
                                 rope_base=wl.rope_base, out=run.dec)
    pre_ms = cold_graph_time_ms(pre, 3, flush)
    dec_ms = cold_graph_time_ms(dec, 10, flush)
    flops = proj_flops(wl, wl.batch * wl.prefill)
    r = wl.rank
    dec_bytes = (codes.nbytes + absmax.nbytes + 2 * (3 * r * wl.d_in + r * wl.n_out)
                 + 2 * wl.batch * (wl.d_in + wl.n_out))
    return {"prefill": {"mean_ms": round(pre_ms, 4), "rows": wl.batch * wl.prefill,
                        "achieved": round(flops / pre_ms / 1e9, 3), "unit": "TFLOP/s",
                        "frac": round(flops / pre_ms / 1e9 / peaks["bf16_tflops_sustained"], 4)},
            "decode": {"mean_ms": round(dec_ms, 5), "rows": wl.batch,
                       "algorithmic_bytes": dec_bytes,
                       "achieved": round(dec_bytes / dec_ms / 1e6, 3), "unit": "GB/s",
                       "frac": round(dec_bytes / dec_ms / 1e6 / peaks["hbm_gbs"], 4)},
            "l2": "flushed before each timed launch"}


def paged_decode_rates(run, peaks, flush):
    """Decode attention over a PAGED cache (256-token pages from one pool, each
    sequence at its own length: continuous batching) with the workload's head
    shape, batch and bit width, lengths spread evenly over [P/2, P] for a
    P-token prefill.  The workload's own format when a paged cache supports it
    (affine, symmetric, KIVI), otherwise an affine cache of the same bit width
    (KVarN caches are uniform only).  Against HBM: every sequence's coded and
    full-precision tokens' bytes plus q and out."""
    from paper_2609_04263_gb300 import kvq
    wl, api = run.wl, run.api
    if wl.dtype != "bf16" or wl.head_dim not in (64, 128) or wl.key_bits not in (2, 4):
        return None
    own = wl.fmt in (synth.FMT_AFFINE, synth.FMT_SYMMETRIC, synth.FMT_KIVI)
    fmt = wl.fmt if own else synth.FMT_AFFINE
    B, H, Hq, D, P = wl.batch, wl.n_kv_heads, wl.n_q_heads, wl.head_dim, wl.prefill
    lens = [P // 2 + (P - P // 2) * b // max(B - 1, 1) for b in range(B)]
    pages = sum((t + 256) // 256 for t in lens)
    desc = api.make_desc(fmt, wl.key_bits, wl.key_bits, 32, B, H, Hq, D, P + 64, torch.bfloat16,
                         residual_tokens=wl.residual_tokens if own else 0,
                         layout=kvq.KVQ_LAYOUT_PAGED, num_pages=pages)
    cache = api.Cache(desc, device=run.dev)
    g = torch.Generator(device="cpu").manual_seed(3)
    for lo in range(0, P, 1024):               # ragged prefill in chunks
        n = [max(0, min(1024, t - lo)) for t in lens]
        L = max(n)
        if L == 0:
            break
        k = torch.randn(B, H, L, D, generator=g).to(torch.bfloat16).to(run.dev)
        v = torch.randn(B, H, L, D, generator=g).to(torch.bfloat16).to(run.dev)
        cache.append_ragged(k, v, n)
    q = torch.randn(B, Hq, 1, D, generator=g).to(torch.bfloat16).to(run.dev)
    out = torch.empty_like(q)
    ms = cold_graph_time_ms(lambda: cache.attend_decode(q, out=out), 10, flush)
    if own:                                    # the workload's format: its own byte count
        nbytes = H * sum(cache_read_bytes(wl, t) for t in lens) + 2 * B * Hq * D * 2
    else:
        per_tok = D * wl.key_bits // 8 * 2 + 2 * (D // 32) * 4
        nbytes = H * per_tok * sum(lens) + 2 * B * Hq * D * 2
    return {"format": {synth.FMT_AFFINE: "affine", synth.FMT_SYMMETRIC: "symmetric",
                       synth.FMT_KIVI: "kivi"}[fmt],
            "bits": wl.key_bits, "sequences": B, "tokens_min": min(lens), "tokens_max": max(lens),
            "pages": pages, "mean_ms": round(ms, 5), "algorithmic_bytes": nbytes,
            "achieved": round(nbytes / ms / 1e6, 3), "unit": "GB/s",
            "frac": round(nbytes / ms / 1e6 / peaks["hbm_gbs"], 4),
            "kernel": "the decode of a uniform cache of this shape, runs of blocks inside one page",
            "l2": "flushed before each timed launch"}


# fp32 FMA rate of the GB300: 152 SMs x 128 fp32 lanes x 2 flops x 2070 MHz
FP32_FMA_TFLOPS = 152 * 128 * 2 * 2.070e9 / 1e12


def ste_backward_rates(run, peaks, flush, max_len=2048):
    """The straight-through backward of one layer (kvq_attend_backward, then
    kvq_lora_backward with d_x) for one sequence of min(prefill, 2048) tokens
    of the workload's shape and cache format: the adapter-training step.  The
    attention products run on fp32 SIMT GEMMs (rated against the fp32 FMA
    rate); with bf16 activations the adapters' dominant product, d_x = g W,
    runs on the tensor cores (rated against the sustained bf16 peak).  None for
    KVarN caches (no backward)."""
    from paper_2609_04263_gb300 import kvq
    wl, api = run.wl, run.api
    if wl.fmt == synth.FMT_KVARN:
        return None
    L, D, Hq, Hkv, d_in, r = min(wl.prefill, max_len), wl.head_dim, wl.n_q_heads, \
        wl.n_kv_heads, wl.d_in, wl.rank
    dev, dt = run.dev, run.dt
    desc = api.make_desc(wl.fmt, wl.key_bits, wl.value_bits, wl.group_size, 1, Hkv, Hq, D, L,
                         dt, residual_tokens=wl.residual_tokens)
    cache = api.Cache(desc, device=dev)
    x = run.x_pre[:1, :L].contiguous()
    w, lora = run.layers[0]
    q, k, v = api.project_lora(x, w, lora, wl.alpha_over_r, Hq, Hkv, D, rope_base=wl.rope_base)
    cache.append(k, v)
    g = torch.Generator(device="cpu").manual_seed(7)
    d_out = torch.randn(q.shape, generator=g).to(dt).to(dev)
    f32 = dict(dtype=torch.float32, device=dev)
    dq, dk, dv = torch.empty(1, Hq, L, D, **f32), torch.empty(1, Hkv, L, D, **f32), \
        torch.empty(1, Hkv, L, D, **f32)
    ws_bytes = kvq.kvq_attend_backward_workspace(cache.handle, L, Hq) * Hkv
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    lws_bytes = kvq.kvq_lora_backward_workspace(1, L, d_in, Hq, Hkv, D, r, r, r)
    lws = torch.empty(lws_bytes, dtype=torch.uint8, device=dev)
    grads = [torch.empty(lora[p][i].shape, **f32) for p in "qkv" for i in (0, 1)]
    dx = torch.empty(1, L, d_in, **f32)
    scale = 1.0 / math.sqrt(D)
    ptr = lambda t: t.data_ptr()

    def attn():
        kvq.kvq_attend_backward(cache.handle, ptr(q), ptr(d_out), L, Hq, scale, ptr(dq),
                                ptr(dk), ptr(dv), ptr(ws), ws_bytes,
                                torch.cuda.current_stream().cuda_stream)

    def adapters():
        fac = [a for p in "qkv" for a in (ptr(lora[p][0]), ptr(lora[p][1]), r)]
        kvq.kvq_lora_backward(ptr(x), 1, L, d_in, ptr(w), *fac, wl.alpha_over_r, Hq, Hkv, D, 0,
                              wl.rope_base, 1 if dt == torch.bfloat16 else 0, ptr(dq), ptr(dk),
                              ptr(dv), L, *[ptr(t) for t in grads], ptr(dx), ptr(lws),
                              lws_bytes, torch.cuda.current_stream().cuda_stream)
    att_ms = cold_graph_time_ms(attn, 3, flush)
    lora_ms = cold_graph_time_ms(adapters, 3, flush)
    visible = L * (L + 1) // 2
    att_flops = 10 * D * Hq * visible             # S, dP, dQ, dK, dV: 2 D per visible pair
    n_out = (Hq + 2 * Hkv) * D
    lora_flops = (2 * L * d_in * 3 * r + 2 * 2 * L * r * n_out + 2 * L * r * 3 * d_in
                  + 2 * L * n_out * d_in + 2 * L * 3 * r * d_in)
    rate = lambda f, ms: round(f / ms / 1e9, 3)
    fma = {"bound": "alu", "value": round(FP32_FMA_TFLOPS, 2), "unit": "TFLOP/s",
           "what": "fp32 FMA: 152 SMs x 128 lanes x 2 flops x 2070 MHz"}
    tensor = dt == torch.bfloat16 and d_in % 128 == 0 and n_out % 64 == 0
    lpeak = ({"bound": "tensor", "value": peaks["bf16_tflops_sustained"], "unit": "TFLOP/s",
              "what": "measured sustained bf16 (d_x = g W as bf16 high + low parts of g: "
                      "twice the algorithmic MMA work)"} if tensor else fma)
    return {"tokens": L, "sequences": 1,
            "attention": {"mean_ms": round(att_ms, 4), "flops": att_flops,
                          "achieved": rate(att_flops, att_ms), "unit": "TFLOP/s",
                          "frac": round(att_flops / att_ms / 1e9 / fma["value"], 4), "peak": fma},
            "adapters": {"mean_ms": round(lora_ms, 4), "flops": lora_flops,
                         "achieved": rate(lora_flops, lora_ms), "unit": "TFLOP/s",
                         "frac": round(lora_flops / lora_ms / 1e9 / lpeak["value"], 4),
                         "peak": lpeak},
            "l2": "flushed before each timed launch"}


# ---------------------------------------------------------------------------
# CPU oracle (the reported baseline and the reference arm)
# ---------------------------------------------------------------------------
def oracle_sample(wl, decode_steps=8, prefill=None, max_queries=64):
    """Time the CPU oracle on one layer of one sequence: a full-length prefill
    (projection, pack, attention) and `decode_steps` decode steps.  Returns
    (seconds, job-equivalent tokens/s, description): the per-layer-per-sequence
    cost is scaled to all layers and sequences and the decode steps to the
    full count (decode steps cost the same to within the cache growth).

    When the prefill has more than `max_queries` tokens, the prefill attention
    runs the oracle's plain attention for `max_queries` evenly spaced queries
    over every key they see (a full [Hq, P, P] fp64 score tensor would not fit
    in host memory at P = 8192), and its time is scaled by the ratio of
    visible (query, key) pairs of all P queries to those of the sample."""
    from oracle import kvq_oracle as O
    P = wl.prefill if prefill is None else prefill
    w, lora = synth.layer_weights(wl, 0)
    act = wl.dtype
    w = O.round_to(w, act)
    lora = {p: tuple(O.round_to(t, act) for t in lora[p]) for p in "qkv"}
    x_pre = O.round_to(synth.hidden_states((1, P, wl.d_in), wl.hidden, wl.outlier_frac), act)
    x_dec = O.round_to(synth.hidden_states((1, decode_steps, wl.d_in), wl.hidden,
                                           wl.outlier_frac, stream=1), act)
    cache = O.OracleCache(wl.fmt, wl.key_bits, wl.value_bits, wl.group_size, 1, wl.n_kv_heads,
                          wl.head_dim, P + decode_steps, act=act,
                          residual_tokens=wl.residual_tokens, sink_tokens=wl.sink_tokens,
                          norm_iters=wl.norm_iters)
    args = (wl.alpha_over_r, wl.n_q_heads, wl.n_kv_heads, wl.head_dim)
    nq = min(P, max_queries)
    ls = np.unique(np.linspace(0, P - 1, nq).round().astype(np.int64))
    t0 = time.perf_counter()
    q, k, v = O.project_lora(x_pre, w, lora, *args, pos0=0, rope_base=wl.rope_base)
    cache.append(O.round_to(k, act), O.round_to(v, act))
    t1 = time.perf_counter()
    if len(ls) == P:
        O.attend(cache, O.round_to(q, act))
        attn_scale = 1.0
    else:
        kh, vh = cache.reconstruct()
        O.attention(O.round_to(q[:, :, ls], act), kh, vh, ls, 1.0 / math.sqrt(wl.head_dim))
        attn_scale = (P * (P + 1) / 2) / float((ls + 1).sum())
    t2 = time.perf_counter()
    for s in range(decode_steps):
        q, k, v = O.project_lora(x_dec[:, s:s + 1], w, lora, *args, pos0=P + s,
                                 rope_base=wl.rope_base)
        cache.append(O.round_to(k, act), O.round_to(v, act))
        O.attend(cache, O.round_to(q, act))
    t3 = time.perf_counter()
    prefill_s = (t1 - t0) + (t2 - t1) * attn_scale
    job_s = (prefill_s + (t3 - t2) * wl.decode / decode_steps) * wl.layers * wl.batch
    tokens = wl.batch * (wl.prefill + wl.decode)
    attn = ("" if len(ls) == P else
            f" (prefill attention of {len(ls)} evenly spaced queries over all their keys, "
            f"scaled by visible pairs x{attn_scale:.1f})")
    return t3 - t0, tokens / job_s, (f"1 of {wl.layers} layers x 1 of {wl.batch} sequences: "
                                     f"{P}-token prefill{attn} + {decode_steps} of {wl.decode} "
                                     f"decode steps, scaled to the full job")


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


# ---------------------------------------------------------------------------
def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, x):
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64,
                     device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def workload_config(wl, world):
    """The `config` object of the JSON line (both arms)."""
    return {
        "workload": wl.name, "layers": wl.layers, "batch": wl.batch,
        "prefill": wl.prefill, "decode": wl.decode, "d_in": wl.d_in,
        "q_heads": wl.n_q_heads, "kv_heads": wl.n_kv_heads, "head_dim": wl.head_dim,
        "cache": f"{synth.FMT_NAMES[wl.fmt]} K{wl.key_bits}V{wl.value_bits} G{wl.group_size}",
        "lora_rank": wl.rank, "tokens_per_step": wl.batch * (wl.prefill + wl.decode),
        "l2": "flushed between timed steps (256 MiB written, then 256 MiB read so no dirty "
              "line is left); job working set > L2",
        "parallelism": f"replicas x{world}",
    }


def run_reference(args, world, rank):
    if rank != 0:
        return
    wl = synth.WORKLOADS[args.workload]
    vals, secs = [], []
    for _ in range(args.warmup):
        oracle_sample(wl, decode_steps=2, prefill=min(wl.prefill, 1024))
    sample = None
    for _ in range(args.steps):
        s, v, sample = oracle_sample(wl, decode_steps=4)
        vals.append(v)
        secs.append(s)
    value = statistics.mean(vals)
    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * wl.batch * (wl.prefill + wl.decode) / value,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": dict(workload_config(wl, world), decode_path="CPU oracle"),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cpu_cores(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="kvq", choices=["kvq", "reference"])
    ap.add_argument("--workload", default=WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    # smaller runs for profiler launch lists (not for reported numbers)
    ap.add_argument("--decode-steps", type=int, default=None,
                    help="decode steps per job (default: the workload's)")
    ap.add_argument("--prefill", type=int, default=None,
                    help="prefill tokens per sequence (default: the workload's)")
    ap.add_argument("--layers", type=int, default=None,
                    help="attention layers (default: the workload's)")
    ap.add_argument("--eager-decode", action="store_true",
                    help="launch decode steps directly instead of replaying a graph")
    ap.add_argument("--separate-decode", action="store_true",
                    help="decode through the three separate calls, not kvq_decode_step")
    ap.add_argument("--timed-only", action="store_true",
                    help="skip the per-kernel, end-to-end and CPU passes")
    args = ap.parse_args()
    world, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank)
        return
    if not torch.cuda.is_available():
        raise SystemExit("bench.py --impl kvq needs a CUDA GPU")
    from paper_2609_04263_gb300 import build
    if rank == 0 or world == 1:
        build.build()
    barrier(world)
    device = f"cuda:{local}"
    torch.cuda.set_device(device)
    wl = synth.WORKLOADS[args.workload]
    import dataclasses
    if args.decode_steps is not None:
        wl = dataclasses.replace(wl, decode=args.decode_steps)
    if args.layers is not None:
        wl = dataclasses.replace(wl, layers=args.layers)
    if args.prefill is not None:
        wl = dataclasses.replace(wl, prefill=args.prefill)
    peaks, peak_kind = load_peaks()
    run = Runner(wl, device)
    run.eager = args.eager_decode
    run.separate = args.separate_decode
    if not run.eager:
        run.capture()
    flush = torch.zeros(512 * 1024 * 1024, dtype=torch.uint8, device=device)

    for _ in range(max(args.warmup, 3)):
        run.job()
    torch.cuda.synchronize()

    # ---- timed region: K whole-job steps, L2 flushed between steps --------
    clocks = ClockSampler(local)
    clocks.start()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    for s in range(args.steps):
        l2_flush(flush)
        run.job(ev[s])
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall
    barrier(world)
    clk = clocks.stop()
    # a bounded wait that gave up inside a kernel returns early with wrong
    # output and would time as a fast step: no value is reported then
    from paper_2609_04263_gb300 import kvq
    status = kvq.kvq_device_status(torch.cuda.current_stream().cuda_stream)
    status = int(max_over_ranks(world, float(status)))
    if status:
        if rank == 0:
            print(json.dumps({"metric": METRIC, "value": None, "unit": "tokens/s",
                              "n_gpus": world, "device_status": status,
                              "error": "a bounded device-side wait gave up during the timed "
                                       "region: the timed output is not valid"}), flush=True)
        raise SystemExit(1)
    step_ms = [e[0].elapsed_time(e[2]) for e in ev]
    pre_ms = [e[0].elapsed_time(e[1]) for e in ev]
    dec_ms = [e[1].elapsed_time(e[2]) for e in ev]
    total_s = max_over_ranks(world, sum(step_ms) / 1000.0)
    tokens_per_step = wl.batch * (wl.prefill + wl.decode)
    value = world * tokens_per_step * args.steps / total_s
    decode_tps = wl.batch * wl.decode / (statistics.mean(dec_ms) / 1000.0)

    if args.timed_only:
        if rank == 0:
            print(json.dumps({"timed_only": True, "ms_per_step": statistics.mean(step_ms),
                              "workload": wl.name, "decode": wl.decode,
                              "eager_decode": run.eager, "decode_path": run.decode_path()}),
              flush=True)
        return

    # ---- per-kernel durations ---------------------------------------------
    # Prefill kernels run for milliseconds: CUDA events around each eager
    # call.  Decode kernels run for microseconds, so each class (projection,
    # append, attention) is captured as a graph of its 22 per-layer calls and
    # timed over repeated replays; the graph keeps the device busy, so the
    # events measure kernel time, not host launch gaps.
    timer = EventTimer()
    run.reset()
    run.prefill(timer)
    mean_ms = timer.mean_ms()
    run.xs.copy_(run.x_dec[0])
    # each decode graph replay appends one token per layer: two untimed
    # replays and `reps` timed ones must fit the cache's decode room
    reps = min(10, wl.decode - 2)
    if reps < 1:
        raise SystemExit("bench.py: the per-kernel timing needs --decode-steps >= 3 "
                         "(or --timed-only)")
    n_dec = wl.layers * wl.decode
    work = {
        "project": ("tensor", proj_flops(wl, wl.batch * wl.prefill), wl.layers),
        "attend_prefill": ("tensor", prefill_attn_flops(wl, wl.prefill, wl.prefill), wl.layers),
        "append": ("hbm", pack_bytes(wl, wl.prefill), wl.layers),
    }
    if run.fused_append:
        # the projection kernel also codes the keys and values: no separate append
        del work["append"]
    if run.separate:
        for name, fn in (("project_decode", run.decode_project_layers),
                         ("append_decode", run.decode_append_layers),
                         ("attend_decode", run.decode_attend_layers)):
            mean_ms[name] = graph_time_ms(fn, reps) / wl.layers
        T_dec = wl.prefill + 2 + reps          # cache length during the attention replays
        work["project_decode"] = ("hbm", proj_bytes(wl, wl.batch), n_dec)
        work["append_decode"] = ("hbm", pack_bytes(wl, 1), n_dec)
        work["attend_decode"] = ("hbm", decode_attn_bytes(wl, T_dec), n_dec)
    else:
        mean_ms["decode_step"] = graph_time_ms(run.decode_step_layers, reps) / wl.layers
        T_dec = wl.prefill + 2 + reps // 2     # mean cache length over the timed replays
        work["decode_step"] = ("hbm", decode_step_bytes(wl, T_dec), n_dec)
    # the packed-cache decode attention alone (kvq_attend_decode over every
    # layer's cache, L2 flushed before each timed replay), against HBM
    att_ms = cold_graph_time_ms(run.decode_attend_layers, reps, flush) / wl.layers
    T_att = run.caches[0].sync()
    att_bytes = decode_attn_bytes(wl, T_att)
    att_rate = att_bytes / (att_ms / 1000.0) / 1e9
    decode_attention = {"mean_ms": round(att_ms, 5), "tokens": T_att,
                        "algorithmic_bytes": att_bytes, "achieved": round(att_rate, 3),
                        "unit": "GB/s", "frac": round(att_rate / peaks["hbm_gbs"], 4),
                        "l2": "flushed before each replay of all layers' calls",
                        "traffic": measured_traffic(wl.name, "decode_attention")}
    nf4 = nf4_projection_rates(run, peaks, flush) if wl.dtype == "bf16" else None
    ste = ste_backward_rates(run, peaks, flush)
    paged = paged_decode_rates(run, peaks, flush)
    share = {k: mean_ms[k] * work[k][2] for k in work}
    dominant = max(share, key=share.get)
    bound, amount, _ = work[dominant]
    dur_s = mean_ms[dominant] / 1000.0
    if bound == "tensor":
        achieved = amount / dur_s / 1e12
        peak = peaks["bf16_tflops_sustained"]
        unit = "TFLOP/s"
    else:
        achieved = amount / dur_s / 1e9
        peak = peaks["hbm_gbs"]
        unit = "GB/s"
    kernels = {}
    for k, (b, amt, n) in work.items():
        d = mean_ms[k] / 1000.0
        rate = amt / d / (1e12 if b == "tensor" else 1e9)
        pk = peaks["bf16_tflops_sustained"] if b == "tensor" else peaks["hbm_gbs"]
        kernels[k] = {"mean_ms": round(mean_ms[k], 5), "launches_per_step": n,
                      "ms_per_step": round(mean_ms[k] * n, 3),
                      "achieved": round(rate, 3), "unit": "TFLOP/s" if b == "tensor" else "GB/s",
                      "frac": round(rate / pk, 4)}

    # ---- end to end through the public API with host buffers --------------
    e2e_vals = []
    o_host = torch.empty(run.o_pre.shape, dtype=run.dt, pin_memory=True)
    od_host = torch.empty(run.o_dec.shape, dtype=run.dt, pin_memory=True)
    h2d = run.x_pre_host.numel() * run.x_pre_host.element_size() + \
        run.x_dec_host.numel() * run.x_dec_host.element_size()
    d2h = o_host.numel() * o_host.element_size() + od_host.numel() * od_host.element_size()
    copy_stream = torch.cuda.Stream()
    # untimed passes first, as for the device-timed steps: the first copies
    # between these pinned buffers and the device run far slower (106 ms
    # instead of 43 ms for the 1 GB prefill input on the 8B-shaped job)
    for _ in range(min(args.warmup, 2)):
        run.job_e2e(run.x_pre_host, run.x_dec_host, o_host, od_host, copy_stream)
    torch.cuda.synchronize()
    for s in range(args.steps):
        l2_flush(flush)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        run.job_e2e(run.x_pre_host, run.x_dec_host, o_host, od_host, copy_stream)
        torch.cuda.synchronize()
        e2e_vals.append(time.perf_counter() - t0)
    e2e_s = max_over_ranks(world, statistics.mean(e2e_vals))
    status = int(max_over_ranks(world, float(
        kvq.kvq_device_status(torch.cuda.current_stream().cuda_stream))))
    e2e_value = world * tokens_per_step / e2e_s

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        secs, cval, sample = oracle_sample(wl, decode_steps=8)
        if secs < 10.0:   # grow the sample toward ~15 s of CPU work on fast hosts
            f = min(8.0, 15.0 / max(secs, 0.5))
            secs, cval, sample = oracle_sample(
                wl, decode_steps=min(wl.decode, int(8 * f)),
                max_queries=min(wl.prefill, int(64 * f)))
        cpu = {"value": cval, "unit": "tokens/s", "cores": cpu_cores(), "kind": "oracle",
               "sample": sample + f" ({secs:.1f} s of CPU time)"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": max(args.warmup, 3),
            "ms_per_step": statistics.mean(step_ms), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
            "config": dict(workload_config(wl, world), decode_path=run.decode_path()),
            "phases": {"prefill_ms": statistics.mean(pre_ms), "decode_ms": statistics.mean(dec_ms),
                       "decode_tokens_per_s": decode_tps,
                       "pack_gbs": kernels["append"]["achieved"] if "append" in kernels else None,
                       "prefill_append": ("fused into the projection (kvq_project_append)"
                                          if run.fused_append else "separate kvq_append_pack"),
                       "qkv_tflops": kernels["project"]["achieved"]},
            "roofline": {"bound": bound, "kernel": dominant, "achieved": round(achieved, 3),
                         "peak": peak, "unit": unit, "frac": round(achieved / peak, 4),
                         "peak_source": f"{peak_kind} "
                                        f"({'bf16_tflops_sustained' if bound == 'tensor' else 'hbm_gbs'})",
                         "traffic": measured_traffic(
                             wl.name, dominant,
                             run.traffic_variant() if dominant == "decode_step" else ""),
                         "algorithmic_bytes" if bound == "hbm" else "algorithmic_flops": amount},
            "kernels": kernels,
            "decode_attention": decode_attention,
            "nf4_projection": nf4,
            "ste_backward": ste,
            "paged_decode": paged,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": run.launches_per_step() * args.steps,
            "device_status": status,
            "clocks": clk,
            "wall_s_timed": t_wall,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
