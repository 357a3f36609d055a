"""Benchmark of the WitCert hot path on GB300: metered decode KV tokens/s,
achieved HBM GB/s against the measured peak, and witness-write GB/s.

One step = one decode step of the workload: for every layer, write the
newest token of every sequence (quantize + witness) and run the metered
decode attention over the whole context; then gate all (layer, sequence,
query head) meters at tau.  The step is captured once in a CUDA graph and
replayed.  Default workload: 28 layers, 28 query / 4 KV heads, head_dim 128,
one sequence of 32768 tokens, dithered INT8 cache, tau = 0.1.

    python bench.py [--gpus N --steps K --warmup W] [--config 1..5] [--impl ours|reference]

Multi-GPU (torchrun): every rank runs its own sequences (different seeds)
with no collective on the data path; a barrier brackets the timed region and
the slowest rank's time is used (weak scaling).
"""

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

BYTES_PER_TOKEN_HEAD = {0: 276, 1: 272}     # decode bytes read per token per KV head
WRITE_BYTES_PER_TOKEN_HEAD = {0: 512 + 276, 1: 512 + 272}
METRIC = "metered decode KV tokens/s & HBM GB/s vs 8 TB/s; witness-write GB/s"


def _traffic(workload):
    """DRAM bytes per decode launch from the committed ncu summary, if the
    kernel source is unchanged since the capture; else None."""
    import hashlib
    try:
        src = open(os.path.join(ROOT, "paper_2607_28699_gb300", "csrc", "decode_kernel.cu"), "rb").read()
        sha = hashlib.sha256(src).hexdigest()[:16]
        for line in open(os.path.join(ROOT, "profiles", "traffic.txt")):
            f = line.split()
            if len(f) == 4 and f[0] == "decode_kernel" and f[1] == sha and f[2] == workload:
                return int(f[3])
    except OSError:
        pass
    return None


def _peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except FileNotFoundError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def barrier(world):
    if world > 1:
        torch.distributed.barrier()


def max_over_ranks(x, world):
    """Largest value over the ranks (the slowest rank's time); the only
    collective, outside the timed region."""
    if world == 1:
        return x
    dev = "cuda" if torch.distributed.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def rank_workload(config, seed, rank):
    """Replicas: every rank runs the same workload shape on its own seeded
    data (no data-path exchange; weak scaling)."""
    return W.config(config, seed=seed + rank)


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def _pack(tensors, align=256):
    """One uint8 device buffer holding copies of ``tensors`` at ``align``-byte
    offsets; returns (buffer, views of it with the tensors' shapes and values)."""
    offs, n = [], 0
    for t in tensors:
        offs.append(n)
        n = (n + t.numel() * t.element_size() + align - 1) // align * align
    buf = torch.zeros(max(n, align), dtype=torch.uint8, device=tensors[0].device)
    views = []
    for t, o in zip(tensors, offs):
        v = buf[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape)
        v.copy_(t)
        views.append(v)
    return buf, views


class Setup:
    """Caches, queries and the per-step buffers of one workload on one GPU.
    extras: also the value-witness and grouped-scale caches of the §8(f) rows
    (the headline workload only)."""

    def __init__(self, wl, dither_bits=8, extras=True):
        import paper_2607_28699_gb300 as wc
        self.wc, self.wl = wc, wl
        self.desc = wc.CacheDesc(num_q_heads=wl.n_q_heads, num_kv_heads=wl.n_kv_heads,
                                 num_pages=wl.num_pages, scheme=wl.scheme, dither_bits=dither_bits,
                                 seed=wl.seed * 7919 + 1)
        bt = W.block_tables(wl)
        sm = W.slot_mapping(wl, bt)
        self.bt = torch.from_numpy(bt).cuda()
        self.sm = torch.from_numpy(sm).cuda()
        self.ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
        last = np.cumsum(wl.ctx_lens) - 1                       # index of each sequence's newest token
        self.new_slots = self.sm[torch.from_numpy(last).cuda()].contiguous()
        self.caches, self.k_new, self.v_new, self.vcaches, self.gcaches = [], [], [], [], []
        # the grouped-scale cache with the outlier-pair bypass (§6.2.3), pairs calibrated on the prefill
        self.gdesc = dataclasses.replace(self.desc, scheme=wc.SCHEME_DITHER_INT8_G32, dither_bits=8)
        for layer in range(wl.n_layers):
            k, v = W.layer_kv(wl, layer, device="cuda")
            cache = wc.LayerCache.empty(self.desc)
            wc.kv_quantize_witness(self.desc, layer, k, v, self.sm, cache)   # prefill write
            self.caches.append(cache)
            if extras:
                # the same cache viewed with a value witness too (value-side measurement only)
                vc = dataclasses.replace(cache, v_witness=torch.zeros(cache.k_witness.shape[:-1] + (2,),
                                                                      dtype=torch.float16, device="cuda"))
                wc.kv_quantize_witness(self.desc, layer, k, v, self.sm, vc)
                self.vcaches.append(vc)
                gc = wc.LayerCache.empty(self.gdesc, num_bypass_pairs=self.BYPASS_PAIRS)
                wc.select_bypass_pairs(k, self.BYPASS_PAIRS, self.desc.rope_layout, pairs=gc.bypass_pairs)
                wc.kv_quantize_witness(self.gdesc, layer, k, v, self.sm, gc)
                self.gcaches.append(gc)
            li = torch.from_numpy(last).cuda()
            self.k_new.append(k[li].contiguous())
            self.v_new.append(v[li].contiguous())
            if layer + 1 < wl.n_layers:
                del k, v
        # write-path throughput: the last layer's whole prefill, rewritten
        # (same inputs, same slots) by warm, back-to-back calls replayed as a
        # graph (device time, without the host's launch overhead)
        def write_s(desc, cache, reps=10):
            one = lambda: [wc.kv_quantize_witness(desc, wl.n_layers - 1, k, v, self.sm, cache) for _ in range(reps)]
            return timed_graph_ms(capture(one), 5, 3) / 1e3 / reps
        self.write_call_s = write_s(self.desc, self.caches[-1])
        if extras:
            self.write_v_call_s = write_s(self.desc, self.vcaches[-1])   # the value witness stored too
            self.write_g_call_s = write_s(self.gdesc, self.gcaches[-1])  # the grouped cache's write
        del k, v
        # the step's new tokens as one stacked tensor per side (one copy in the end-to-end step)
        self.k_new_all, self.v_new_all = torch.stack(self.k_new), torch.stack(self.v_new)
        self.k_new, self.v_new = list(self.k_new_all), list(self.v_new_all)
        self.q = torch.stack([W.layer_queries(wl, layer, device="cuda") for layer in range(wl.n_layers)])
        self.ws = wc.Workspace(self.desc, wl.batch, wl.max_pages)
        L, B, Hq = wl.n_layers, wl.batch, wl.n_q_heads
        self.out = torch.empty(L, B, Hq, 128, dtype=torch.float32, device="cuda")
        self.meter = torch.empty(L, B, Hq, dtype=torch.float32, device="cuda")
        self.raw = torch.empty(L, B, Hq, dtype=torch.float32, device="cuda")
        self.keep_q = torch.empty(L * B * Hq, dtype=torch.uint8, device="cuda")
        self.keep_kv = torch.empty(L * B * Hq // wl.group, dtype=torch.uint8, device="cuda")
        self.n_kept = torch.empty(2, dtype=torch.int32, device="cuda")
        self.tau = wl.taus[0]
        # the step's inputs and its read-back results, each set laid out in one
        # buffer (256-byte aligned views), so the end-to-end step moves them with
        # one copy per direction
        self.in_buf, (self.q, self.k_new_all, self.v_new_all, self.ctx) = _pack(
            (self.q, self.k_new_all, self.v_new_all, self.ctx))
        self.k_new, self.v_new = list(self.k_new_all), list(self.v_new_all)
        self.out_buf, (self.out, self.raw, self.meter, self.keep_q, self.n_kept) = _pack(
            (self.out, self.raw, self.meter, self.keep_q, self.n_kept))

    def decode(self, layer):
        self.wc.metered_decode_attention(self.desc, layer, self.q[layer], self.bt, self.ctx, self.caches[layer],
                                         self.ws, out=self.out[layer], meter=self.meter[layer],
                                         meter_raw=self.raw[layer])

    @property
    def fused_append(self):
        """The step writes each new token inside the decode (dithered INT8, 8-bit dither)."""
        return self.wl.scheme == 0 and self.desc.dither_bits == 8

    def step(self):
        wc, wl = self.wc, self.wl
        for layer in range(wl.n_layers):
            if self.fused_append:
                wc.metered_decode_attention_append(
                    self.desc, layer, self.q[layer], self.bt, self.ctx, self.caches[layer], self.ws,
                    self.k_new[layer], self.v_new[layer], self.new_slots, out=self.out[layer],
                    meter=self.meter[layer], meter_raw=self.raw[layer])
            else:
                wc.kv_quantize_witness(self.desc, layer, self.k_new[layer], self.v_new[layer], self.new_slots,
                                       self.caches[layer])
                self.decode(layer)
        wc.gate(self.raw.reshape(-1), wl.group, self.tau, self.keep_q, self.keep_kv, self.n_kept)

    def decode_all(self):
        for layer in range(self.wl.n_layers):
            self.decode(layer)

    def decode_all_value(self):
        """The same calls with the value-side terms and output bound (§3, §4.2)."""
        if not hasattr(self, "vterm"):
            self.vterm, self.vmax, self.obound = (torch.empty_like(self.meter) for _ in range(3))
        for layer in range(self.wl.n_layers):
            self.wc.metered_decode_attention_v(
                self.desc, layer, self.q[layer], self.bt, self.ctx, self.vcaches[layer], self.ws,
                out=self.out[layer], meter=self.meter[layer], meter_raw=self.raw[layer],
                value_term=self.vterm[layer], v_max=self.vmax[layer], out_bound=self.obound[layer])

    TIER_B_DELTA_REQ = 1e-2   # request-level budget, split over layers, query heads and one step
    BYPASS_PAIRS = 4          # m, the paper's default budget (Table "bypassbudget")

    def decode_all_grouped(self, tier_b=False):
        """The same calls over the grouped-scale cache (meters into their own buffers)."""
        wl = self.wl
        if not hasattr(self, "g_raw"):
            self.g_raw, self.g_meter, self.g_b, self.g_b_raw = (torch.empty_like(self.raw) for _ in range(4))
            self.gws = self.wc.Workspace(self.gdesc, wl.batch, wl.max_pages)   # its own split plan
        delta_loc = self.TIER_B_DELTA_REQ / (wl.n_layers * wl.n_q_heads)
        for layer in range(wl.n_layers):
            if tier_b:
                self.wc.metered_decode_attention_tier_b(
                    self.gdesc, layer, self.q[layer], self.bt, self.ctx, self.gcaches[layer], self.gws, delta_loc,
                    out=self.out[layer], meter=self.g_meter[layer], meter_raw=self.g_raw[layer],
                    meter_b=self.g_b[layer], meter_b_raw=self.g_b_raw[layer])
            else:
                self.wc.metered_decode_attention(
                    self.gdesc, layer, self.q[layer], self.bt, self.ctx, self.gcaches[layer], self.gws,
                    out=self.out[layer], meter=self.g_meter[layer], meter_raw=self.g_raw[layer])

    def decode_all_tier_b(self):
        """The same calls with the Tier-B certificate as well (§4.2; dithered INT8 only)."""
        wl = self.wl
        if not hasattr(self, "meter_b"):
            self.meter_b = torch.empty_like(self.meter)
            self.meter_b_raw = torch.empty_like(self.raw)
        delta_loc = self.TIER_B_DELTA_REQ / (wl.n_layers * wl.n_q_heads)
        for layer in range(wl.n_layers):
            self.wc.metered_decode_attention_tier_b(
                self.desc, layer, self.q[layer], self.bt, self.ctx, self.caches[layer], self.ws, delta_loc,
                out=self.out[layer], meter=self.meter[layer], meter_raw=self.raw[layer],
                meter_b=self.meter_b[layer], meter_b_raw=self.meter_b_raw[layer])

    def decode_all_repair(self, select=True):
        """The same calls emitting the per-page meter terms, the gate, then the
        block-level repair selection of every cell the gate flagged (§6.3.5)."""
        wc, wl = self.wc, self.wl
        L, B, Hq = wl.n_layers, wl.batch, wl.n_q_heads
        if not hasattr(self, "page_terms"):
            f32, i32 = dict(dtype=torch.float32, device="cuda"), dict(dtype=torch.int32, device="cuda")
            self.page_terms = torch.empty(L, B, Hq, wl.max_pages, 2, **f32)
            self.softmax_norm = torch.empty(L, B, Hq, 2, **f32)
            self.rep_pages = torch.empty(L, B, Hq, wl.max_pages, **i32)
            self.n_rep = torch.empty(L, B, Hq, **i32)
            self.d_after = torch.empty(L, B, Hq, **f32)
        for layer in range(L):
            wc.metered_decode_attention_repair(
                self.desc, layer, self.q[layer], self.bt, self.ctx, self.caches[layer], self.ws,
                out=self.out[layer], meter=self.meter[layer], meter_raw=self.raw[layer],
                page_terms=self.page_terms[layer], softmax_norm=self.softmax_norm[layer])
        if select:
            wc.gate(self.raw.reshape(-1), wl.group, self.tau, self.keep_q, self.keep_kv, self.n_kept)
            self.select_all()

    def select_all(self):
        """One selection call for the cells of all layers: layers stacked along
        the batch dimension, each row with its sequence's context length."""
        L, B, Hq, P = self.wl.n_layers, self.wl.batch, self.wl.n_q_heads, self.wl.max_pages
        if not hasattr(self, "ctx_rows"):
            self.ctx_rows = self.ctx.repeat(L)
        self.wc.repair_select(self.page_terms.view(L * B, Hq, P, 2), self.softmax_norm.view(L * B, Hq, 2),
                              self.ctx_rows, self.tau, keep_q=self.keep_q, contrib=False,
                              repair_pages=self.rep_pages.view(L * B, Hq, P), n_repair=self.n_rep.view(L * B, Hq),
                              d_after=self.d_after.view(L * B, Hq))

    def launches_per_step(self):
        # per layer: decode kernel (with the new token's write fused) and merge kernel,
        # or write, decode and merge kernels; then one gate
        return (2 if self.fused_append else 3) * self.wl.n_layers + 1

    def decode_bytes_per_launch(self):
        return sum(self.wl.ctx_lens) * self.wl.n_kv_heads * BYTES_PER_TOKEN_HEAD[self.wl.scheme]


def capture(fn):
    """Capture fn into a CUDA graph; replays run on the current stream."""
    g = torch.cuda.CUDAGraph()
    fn()                                       # warm once outside capture (lazy init)
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize()
    return g


def timed_graph_ms(g, steps, warmup):
    """Average ms per replay of a captured graph (events at the graph ends)."""
    for _ in range(warmup):
        g.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(steps):
        g.replay()
    t1.record()
    torch.cuda.synchronize()
    return t0.elapsed_time(t1) / steps


def meter_off_call_ms(st, args):
    """The headline's decode calls through the library built with the
    certificate compiled out of the warp-specialized decode (-DWC_METER_OFF:
    no witness copy, bound MMAs or meter accumulator), for the certificate's
    marginal cost (§8(d) meter on / off).  Outputs go to scratch buffers."""
    import ctypes
    path = os.path.join(ROOT, "paper_2607_28699_gb300", "_lib", "libwitcert_meteroff.so")
    lib = ctypes.CDLL(path)
    vp, i32 = ctypes.c_void_p, ctypes.c_int32
    f = lib.wc_metered_decode_attention
    f.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
    f.restype = ctypes.c_int
    wl, d = st.wl, st.desc.c()
    out, meter, raw = torch.empty_like(st.out[0]), torch.empty_like(st.meter[0]), torch.empty_like(st.raw[0])
    P = lambda t: ctypes.c_void_p(t.data_ptr())

    def calls():
        s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
        for layer in range(wl.n_layers):
            c = st.caches[layer]
            r = f(ctypes.byref(d), layer, P(st.q[layer]), P(st.bt), wl.max_pages, P(st.ctx), wl.batch,
                  P(c.k_codes), P(c.v_codes), P(c.k_scale), P(c.v_scale), P(c.k_witness), P(out), P(meter), P(raw),
                  st.ws.ptr(), st.ws.nbytes, s)
            if r != 0:
                raise RuntimeError(f"meter-off decode failed: {lib.wc_last_error().decode()}")

    return timed_graph_ms(capture(calls), args.steps, args.warmup) / wl.n_layers


def measure_config(cfg, args, world):
    """One of the other workloads, measured like the headline: the step (every
    layer's write + metered decode, then the gate) as a graph, the decode calls
    alone (roofline), the end-to-end step with host copies, and the prefill
    write of one layer."""
    wl = W.config(cfg, seed=args.seed)
    st = Setup(wl, dither_bits=8, extras=False)
    peak = (_peaks() or {}).get("hbm_gbs", 6800.0)
    step_ms = timed_graph_ms(capture(st.step), args.steps, args.warmup)
    dec_ms = timed_graph_ms(capture(st.decode_all), args.steps, args.warmup) / wl.n_layers
    status = st.wc.read_status(st.ws)
    e2e = run_e2e(st, args, world)
    algo = st.decode_bytes_per_launch()
    write_th = sum(wl.ctx_lens) * wl.n_kv_heads
    kept = st.n_kept.cpu().tolist()
    ncell = wl.n_layers * wl.batch * wl.n_q_heads
    gate = {"tau": st.tau, "kept_q_frac": kept[0] / ncell}
    if len(wl.taus) > 1:   # the sweep of taus on the step's meters (risk-ranked gating, §4.3)
        raw = st.raw.reshape(-1)
        gate["kept_q_frac_by_tau"] = {str(t): float((raw <= t).float().mean()) for t in wl.taus}
    res = {"workload": wl.name, "layers": wl.n_layers, "batch": wl.batch, "ctx_tokens": sum(wl.ctx_lens),
           "scheme": "dither-int8" if wl.scheme == 0 else "fp8-e4m3",
           "step": "write of each new token fused into its decode" if st.fused_append else "write kernel, then decode",
           "ms_per_step": step_ms, "kv_tokens_per_s": wl.kv_tokens / (step_ms / 1e3),
           "decode_call_ms": dec_ms, "decode_gbs": algo / (dec_ms / 1e3) / 1e9,
           "frac": algo / (dec_ms / 1e3) / 1e9 / peak, "algorithmic_bytes_per_call": algo,
           "traffic": _traffic(wl.name),
           "e2e": e2e,
           "witness_write_gbs": write_th * WRITE_BYTES_PER_TOKEN_HEAD[wl.scheme] / st.write_call_s / 1e9,
           "gate": gate, "device_status": status,
           "l2": f"inputs {st.caches[0].nbytes() * wl.n_layers / 1e9:.2f} GB per step vs 129 MB L2; no flush"}
    del st
    torch.cuda.empty_cache()
    return res


def run_ours(args, rank, world, local):
    wl = rank_workload(args.config, args.seed, rank)
    if args.layers:
        wl.n_layers = args.layers
    st = Setup(wl, dither_bits=args.dither_bits)
    stream = torch.cuda.current_stream()
    graph = capture(st.step)

    # ---- device-resident timed region ----------------------------------
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    barrier(world)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        torch.cuda.synchronize()
        t0.record(stream)
        for _ in range(args.steps):
            graph.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms = t0.elapsed_time(t1) / args.steps
    ms = max_over_ranks(ms, world)
    status = st.wc.read_status(st.ws)

    # ---- the dominant call alone: all layers' metered decode back to back ----
    # (events only at the ends of the replayed graph, so they do not split it)
    dgraph = capture(st.decode_all)
    for _ in range(args.warmup):
        dgraph.replay()
    torch.cuda.synchronize()
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    d0.record()
    for _ in range(args.steps):
        dgraph.replay()
    d1.record()
    torch.cuda.synchronize()
    dec_avg_ms = d0.elapsed_time(d1) / (args.steps * wl.n_layers)

    # ---- the certificate's marginal cost: the same calls with it compiled out ----
    meter_off = None
    if wl.scheme == 0 and args.dither_bits == 8:
        off_ms = meter_off_call_ms(st, args)
        meter_off = {"decode_call_ms_meter_on": dec_avg_ms, "decode_call_ms_meter_off": off_ms,
                     "certificate_cost": dec_avg_ms / off_ms - 1.0,
                     "build": "libwitcert_meteroff.so (-DWC_METER_OFF): no witness copy, bound MMAs or meter sums"}

    # ---- the same calls with the value side too (its marginal cost) ----
    vgraph = capture(st.decode_all_value)
    for _ in range(args.warmup):
        vgraph.replay()
    torch.cuda.synchronize()
    d0.record()
    for _ in range(args.steps):
        vgraph.replay()
    d1.record()
    torch.cuda.synchronize()
    v_ms = d0.elapsed_time(d1) / (args.steps * wl.n_layers)
    kq, _, _ = st.wc.gate_joint(st.raw.reshape(-1), st.vterm.reshape(-1), st.vmax.reshape(-1), wl.group,
                                st.tau, st.tau)
    value_side = {"decode_call_ms": v_ms, "overhead_vs_plain": v_ms / dec_avg_ms - 1.0,
                  "write_ms_per_layer_prefill": st.write_v_call_s * 1e3,
                  "write_overhead_vs_plain": st.write_v_call_s / st.write_call_s - 1.0,
                  "joint_kept_frac_at_tau": float(kq.float().mean()),
                  "out_bound_median": float(st.obound.median()),
                  "rel_value_term_median": float((st.vterm / st.vmax.clamp_min(1e-30)).median())}

    # ---- the same calls with the Tier-B certificate too (its marginal cost) ----
    tier_b = None
    if wl.scheme == 0:
        bgraph = capture(st.decode_all_tier_b)
        for _ in range(args.warmup):
            bgraph.replay()
        torch.cuda.synchronize()
        d0.record()
        for _ in range(args.steps):
            bgraph.replay()
        d1.record()
        torch.cuda.synchronize()
        tb_ms = d0.elapsed_time(d1) / (args.steps * wl.n_layers)
        mb = st.meter_b_raw.reshape(-1)
        tier_b = {"decode_call_ms": tb_ms, "overhead_vs_tier_a": tb_ms / dec_avg_ms - 1.0,
                  "delta_req": st.TIER_B_DELTA_REQ, "kept_frac_at_tau": float((mb <= st.tau).float().mean()),
                  "meter_b_raw_median": float(mb.median())}

    # ---- the same calls emitting the repair terms, gate, repair selection (§6.3.5) ----
    def graph_ms(fn, per):
        g = capture(fn)
        for _ in range(args.warmup):
            g.replay()
        torch.cuda.synchronize()
        d0.record()
        for _ in range(args.steps):
            g.replay()
        d1.record()
        torch.cuda.synchronize()
        return d0.elapsed_time(d1) / (args.steps * per)

    terms_ms = graph_ms(lambda: st.decode_all_repair(select=False), wl.n_layers)   # decode with the terms
    rep_ms = graph_ms(st.decode_all_repair, wl.n_layers)        # decode + gate + selection, per layer
    sel_ms = graph_ms(st.select_all, wl.n_layers)               # selection alone (one call), per layer
    flag = st.keep_q.view(st.n_rep.shape) == 0
    n_pages = torch.tensor([(c + 15) // 16 for c in wl.ctx_lens], device="cuda").view(1, -1, 1).expand_as(st.n_rep)
    nr = st.n_rep[flag].float()
    repair = {"decode_call_ms": terms_ms, "decode_overhead_vs_plain": terms_ms / dec_avg_ms - 1.0,
              "select_ms_per_layer": sel_ms, "select_launches_per_step": 1,
              "decode_gate_select_ms_per_layer": rep_ms,
              "overhead_vs_plain_decode": rep_ms / dec_avg_ms - 1.0,
              "flagged_cells": int(flag.sum()),
              "pages_per_flagged_cell_median": float(nr.median()) if nr.numel() else 0.0,
              "pages_per_flagged_cell_mean": float(nr.mean()) if nr.numel() else 0.0,
              "page_in_frac_vs_whole_head": float(nr.sum() / n_pages[flag].float().sum()) if nr.numel() else 0.0,
              "d_after_max": float(st.d_after[flag].max()) if nr.numel() else 0.0}

    # ---- the grouped-scale cache with the outlier-pair bypass (§6.2.3) ----------
    g_ms = graph_ms(st.decode_all_grouped, wl.n_layers)
    gb_ms = graph_ms(lambda: st.decode_all_grouped(tier_b=True), wl.n_layers)
    grouped = {"bypass_pairs": st.BYPASS_PAIRS, "decode_call_ms": g_ms, "overhead_vs_plain": g_ms / dec_avg_ms - 1.0,
               "decode_tier_b_call_ms": gb_ms,
               "write_ms_per_layer_prefill": st.write_g_call_s * 1e3,
               "kept_frac_tier_a_at_tau": float((st.g_raw <= st.tau).float().mean()),
               "kept_frac_tier_b_at_tau": float((st.g_b_raw <= st.tau).float().mean()),
               "meter_raw_median": float(st.g_raw.median()), "meter_b_raw_median": float(st.g_b_raw.median()),
               "bytes_per_token_head": st.gcaches[0].nbytes() / (wl.num_pages * 16 * wl.n_kv_heads)}

    kv_tokens_step = wl.kv_tokens
    value = kv_tokens_step * world / (ms / 1e3)
    algo_bytes = st.decode_bytes_per_launch()
    peaks = _peaks() or {}
    peak = peaks.get("hbm_gbs", 6800.0)
    achieved = algo_bytes / (dec_avg_ms / 1e3) / 1e9
    step_gbs = algo_bytes * wl.n_layers / (ms / 1e3) / 1e9

    # ---- end-to-end: host buffers, copies inside the timed region --------
    e2e = run_e2e(st, args, world)

    # ---- write path: one layer's full prefill (all sequences, all KV heads) ----
    write_th = sum(wl.ctx_lens) * wl.n_kv_heads
    write_gbs = write_th * WRITE_BYTES_PER_TOKEN_HEAD[wl.scheme] / st.write_call_s / 1e9

    # ---- gate summary ---------------------------------------------------------
    kept = st.n_kept.cpu().tolist()
    ncell = wl.n_layers * wl.batch * wl.n_q_heads
    coverage = {"tau": st.tau, "kept_q_frac": kept[0] / ncell, "kept_kv_frac": kept[1] / (ncell // wl.group)}
    meters = st.raw.reshape(-1).cpu().numpy()
    coverage["meter_raw_median"] = float(np.median(meters))
    coverage["overflow_cells"] = int(np.sum(~np.isfinite(meters)))

    res = {
        "metric": METRIC, "value": value, "unit": "KV tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int8-dither+fp16-mma/fp32" if wl.scheme == 0 else "fp8-e4m3+fp16-mma/fp32",
        "data": "synthetic (seeded; log-normal outlier channels, 8x sink token, RoPE theta 1e4)",
        "config": {"workload": wl.name, "layers": wl.n_layers, "q_heads": wl.n_q_heads,
                   "kv_heads": wl.n_kv_heads, "head_dim": 128, "batch": wl.batch,
                   "ctx_tokens": sum(wl.ctx_lens), "page": 16, "dither_bits": args.dither_bits,
                   "tau": st.tau, "parallelism": f"replica-per-gpu x{world}",
                   "step": "write of each new token fused into its decode" if st.fused_append
                           else "write kernel, then decode",
                   "l2": f"inputs {st.caches[0].nbytes() * wl.n_layers / 1e9:.2f} GB per step > 129 MB L2; no flush"},
        "hbm_gbs_step": step_gbs,
        "decode_call_ms": dec_avg_ms,
        "meter_off": meter_off,
        "tier_b": tier_b,
        "value_side": value_side,
        "repair": repair,
        "grouped": grouped,
        "roofline": {"kernel": ("decode_ws_kernel" if wl.scheme == 0 and args.dither_bits == 8 else "decode_kernel")
                               + " + merge_kernel (one metered_decode_attention call)",
                     "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": _traffic(wl.name),
                     "frac_of_nominal_8tbs": achieved / 8000.0,
                     "peak_source": "MEASURED_PEAKS.json hbm_gbs (measured copy)" if peaks else "fallback 6.8 TB/s",
                     "algorithmic_bytes_per_launch": algo_bytes},
        "witness_write": {"gbs": write_gbs, "token_heads_per_s": write_th / st.write_call_s,
                          "ms_per_layer_prefill": st.write_call_s * 1e3, "token_heads_per_call": write_th,
                          "bytes_per_token_head": WRITE_BYTES_PER_TOKEN_HEAD[wl.scheme],
                          "frac_of_peak": write_gbs / (_peaks() or {}).get("hbm_gbs", 6800.0)},
        "gate": coverage,
        "gpu_launches": st.launches_per_step() * args.steps,
        "device_status": status,
        "clocks": clk.summary(),
        "e2e": e2e,
    }
    if world == 1 and not args.no_configs:
        # the other workloads, each at its full size on this GPU (not in the headline value)
        st = graph = dgraph = vgraph = bgraph = None   # free the headline's caches and graphs first
        torch.cuda.empty_cache()
        res["configs"] = {f"config{c}": measure_config(c, args, world) for c in range(1, 6) if c != args.config}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline(wl, args)
    return res


def run_e2e(st, args, world):
    """Same step with inputs copied from pinned host memory and results read back."""
    wl = st.wl
    # q, the new K/V rows and the context lengths are views of st.in_buf; out,
    # the meters, the gate's bits and counts views of st.out_buf
    host_in = st.in_buf.cpu().pin_memory()
    host_out = torch.empty_like(st.out_buf, device="cpu").pin_memory()

    def e2e_step():
        st.in_buf.copy_(host_in, non_blocking=True)
        st.step()
        host_out.copy_(st.out_buf, non_blocking=True)

    g = capture(e2e_step)
    for _ in range(max(3, args.warmup)):
        g.replay()
    torch.cuda.synchronize()
    barrier(world)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        g.replay()
    t1.record()
    torch.cuda.synchronize()
    barrier(world)
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, world)
    bi = host_in.numel() * host_in.element_size()      # the copied buffers (with their alignment padding)
    bo = host_out.numel() * host_out.element_size()
    return {"value": wl.kv_tokens * world / (ms / 1e3), "unit": "KV tokens/s", "ms_per_step": ms,
            "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo}


# ---------------------------------------------------------------------------
# oracle legs (CPU)
# ---------------------------------------------------------------------------

def _oracle_layers(wl, layers, budget_s):
    """Time the oracle's decode of the given layers (all KV heads, the first
    one or two sequences) until ``budget_s`` of decode time is spent (at least
    one layer); returns (KV tokens, decode seconds, layers done, sequences).
    Runs in a worker process of the oracle pool; the untimed part is the
    oracle's own write of the cache the decode reads."""
    from oracle import pipeline as OP
    od = OP.Desc(num_q_heads=wl.n_q_heads, num_kv_heads=wl.n_kv_heads, num_pages=wl.num_pages,
                 scheme=wl.scheme, dither_bits=8, seed=wl.seed * 7919 + 1)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    seqs = min(wl.batch, 2)
    n = sum(wl.ctx_lens[:seqs])
    done_tokens, spent, done = 0, 0.0, 0
    for layer in layers:
        if done and spent >= budget_s:
            break
        k, v = W.layer_kv(wl, layer, seq_range=(0, seqs))
        q = W.layer_queries(wl, layer)
        cache = OP.empty_cache(od)
        OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm[:n], cache)
        t = time.perf_counter()
        for b in range(seqs):
            OP.decode_sequence(od, layer, q[b].numpy(), bt[b], wl.ctx_lens[b], cache)
        spent += time.perf_counter() - t
        done_tokens += n
        done += 1
    return done_tokens, spent, done, seqs


class OraclePool:
    """One worker process per host core (spawned: the parent has a CUDA
    context), all timing the oracle at once; a round's value is the sum of the
    workers' KV tokens per decode-second."""

    def __init__(self, workers=None):
        import multiprocessing as mp
        self.workers = workers or os.cpu_count() or 1
        self.pool = mp.get_context("spawn").Pool(self.workers)

    def round(self, wl, budget_s, first_layer=0, layers_each=1):
        jobs = [(wl, [(first_layer + w + j * self.workers) % wl.n_layers for j in range(layers_each)], budget_s)
                for w in range(self.workers)]
        res = self.pool.starmap(_oracle_layers, jobs)
        rate = sum(t / s for t, s, _, _ in res if s > 0)
        tokens, layers, seqs = sum(r[0] for r in res), sum(r[2] for r in res), res[0][3]
        secs = max(r[1] for r in res)
        return rate, (f"{self.workers} processes at once, each the oracle's decode of layers x {seqs} sequence(s) "
                      f"x all KV heads: {layers} layer decodes, {tokens} KV tokens, up to {secs:.3g} s each")

    def close(self):
        self.pool.close()
        self.pool.join()


def cpu_baseline(wl, args):
    pool = OraclePool()
    try:
        layers_each = max(1, -(-wl.n_layers // pool.workers))   # every layer at least once over the pool
        tok_s, sample = pool.round(wl, args.cpu_budget, 0, layers_each)
    finally:
        pool.close()
    return {"value": tok_s, "unit": "KV tokens/s", "cores": pool.workers, "kind": "oracle", "sample": sample,
            "host_cores_available": os.cpu_count()}


def run_reference(args, rank, world):
    if rank != 0:
        return None
    wl = W.config(args.config, seed=args.seed)
    pool = OraclePool()
    try:
        for i in range(args.warmup):
            pool.round(wl, 0.0, i)
        per_step, sample = [], ""
        for i in range(args.steps):
            tok_s, sample = pool.round(wl, args.cpu_budget / max(args.steps, 1), args.warmup + i)
            per_step.append(tok_s)
    finally:
        pool.close()
    value = statistics.median(per_step)
    ms = wl.kv_tokens / value * 1e3
    return {"metric": METRIC, "value": value, "unit": "KV tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)", "impl": "reference",
            "config": {"workload": wl.name, "parallelism": f"{pool.workers} CPU processes (oracle)"},
            "cpu_baseline": {"value": value, "unit": "KV tokens/s", "cores": pool.workers, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "KV tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--layers", type=int, default=0, help="override the layer count (profiling only)")
    ap.add_argument("--dither-bits", type=int, default=8)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the other workloads' measurements")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank, world, local = dist_env()
    if args.impl == "reference":
        res = run_reference(args, rank, world)
        if res is not None:
            print(json.dumps(res))
        return
    torch.cuda.set_device(local)
    if world > 1:
        torch.distributed.init_process_group("nccl")
    res = run_ours(args, rank, world, local)
    if rank == 0:
        print(json.dumps(res))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
