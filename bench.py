#!/usr/bin/env python
"""Benchmark of the routed block (score -> top-K -> gather -> pruned SwiGLU FFN
-> scatter-add) on GB300, one JSON line on stdout (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config long_7b] [--quick]
  python bench.py --impl reference ...      # the CPU oracle on the same workload
  python bench.py --sweep                   # the 7B sweep grid, one line per point

A step is one cer_routed_block call (in place on the residual stream h) over
the whole synthetic batch of the workload, inputs resident in HBM.  The
headline workload is the largest config, long_7b (B = 2, N = 4096, d = 3584);
the line also carries the other full-size configs (und_1p5b, gen_1p5b) and a
summary of the whole 7B sweep grid, each stage against its roofline.  Between
timed steps, outside the timed interval, h is restored from a pristine copy
and L2 is flushed (a 256 MiB write); each step is timed with CUDA events on
the launching stream.  For N > 1 each
rank runs its own replica batch (weak scaling, no data-path collective); the
slowest rank's time is reported.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2608_29291_gb300 import inputs as gen  # noqa: E402
from paper_2608_29291_gb300 import runtime  # noqa: E402

METRIC = "routed block tokens/s; FFN TFLOP/s & gather/scatter GB/s vs GB300 peak"
UNIT = "tokens/s"
# launches per step: [time-bias table (generation only)], scorer GEMM, top-K,
# row gather, gate/up GEMM, down GEMM
def kernels_per_step(task: int) -> int:
    return 6 if task == 1 else 5
FLUSH_BYTES = 256 << 20   # > 129 MB L2
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
GEMM_SOURCES = ("ffn_kernel.cu", "umma_gemm.cuh", "ptx.cuh")


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def gemm_source_hash() -> str:
    h = hashlib.sha256()
    for name in GEMM_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_29291_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str):
    """DRAM bytes per gate/up launch from a committed ncu summary
    (profiles/ffn_gateup_*.md) taken on this workload with the current kernel
    sources; None if there is none."""
    import glob
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "ffn_gateup_*.md"))):
        text = open(path).read()
        m_src = re.search(r"kernel_source_hash:\s*([0-9a-f]+)", text)
        m_wl = re.search(r"workload:\s*(\S+)", text)
        m_b = re.search(r"dram_bytes_per_launch:\s*([0-9]+)", text)
        if m_src and m_wl and m_b and m_src.group(1) == gemm_source_hash() and m_wl.group(1) == workload:
            return int(m_b.group(1))
    return None


class ClockSampler:
    """nvidia-smi clock / throttle sampling around the timed region."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        self.t0 = time.time()

    def stop(self):
        if self.proc is None:
            return
        time.sleep(0.05)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        self.lines = [ln for ln in out.splitlines() if ln.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def smi_index(local_rank: int) -> str:
    """nvidia-smi's name for this rank's GPU (honours CUDA_VISIBLE_DEVICES)."""
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [x.strip() for x in vis.split(",") if x.strip()]
        if local_rank < len(ids):
            return ids[local_rank]
    return str(local_rank)


def workload_config(w: gen.Workload, flush: bool) -> dict:
    return {"workload": w.name, "B": w.B, "N": w.N, "d": w.d, "intermediate": w.I, "kept_channels": w.C,
            "routable": [w.r0, w.r1], "K": w.K, "kept_rows": w.M, "core_hidden": w.Hc, "exp_hidden": w.He,
            "task": "generation" if w.task == 1 else "understanding",
            "l2": "flushed between timed steps (256 MiB write)" if flush else "not flushed",
            "inputs": "seeded synthetic (SplitMix64 normals), resident in HBM"}


def device_time(torch, stream, flush, fn, reps=20):
    """Mean device time (ms) of fn's launches after 3 untimed calls, L2
    flushed before each; a GPU spin before the start event keeps the host's
    launch overhead out of the interval."""
    ms = []
    for i in range(reps + 3):
        flush.fill_(float(i))
        torch.cuda._sleep(200000)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        b.synchronize()
        if i >= 3:
            ms.append(a.elapsed_time(b))
    return float(np.mean(ms))


def measure_attention(cer, torch, w, flush, stream, dev, peak_tf, reps=20):
    """Rotary embedding and attention over the packed sequences (L = k_tot
    retained tokens per sequence) with the workload's backbone heads: causal
    for understanding (prefill), bidirectional for generation.  Synthetic
    packed rows; positions are an ascending keep list."""
    Hq, Hkv = w.attn_heads()
    L = w.k_tot
    causal = 1 if w.task == 0 else 0
    width = (Hq + 2 * Hkv) * 128
    bits = gen.bf16_normal(w.seed, "attn_qkv", (w.B * L, width), 1.0)
    qkv0 = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(dev)
    qkv = qkv0.clone()
    rng = np.random.default_rng(w.seed)
    pos = np.concatenate([np.sort(rng.choice(w.N, L, replace=False)) for _ in range(w.B)]).astype(np.int32)
    pos_d = torch.from_numpy(pos).to(dev)
    out = torch.empty((w.B * L, Hq * 128), dtype=torch.bfloat16, device=dev)
    t_rope = device_time(torch, stream, flush, lambda: cer.cer_rope_packed(qkv, w.B, L, Hq, Hkv, pos_d, 1e6,
                                                                          stream=stream), reps)
    t_attn = device_time(torch, stream, flush, lambda: cer.cer_packed_attention(qkv, w.B, L, Hq, Hkv, causal, out,
                                                                               stream=stream), reps)
    # The whole sublayer from the residual stream: pack, QKV projection, rotary
    # embedding, attention, output projection with the scatter-add.
    h = torch.from_numpy(gen.bf16_normal(w.seed, "attn_h", (w.B, w.N, w.d), 1.0).view(np.int16)).view(
        torch.bfloat16).to(dev)
    hout = torch.empty_like(h)
    WqkvT = torch.from_numpy(gen.bf16_normal(w.seed, "wqkv", (w.d, width), w.d ** -0.5).view(np.int16)).view(
        torch.bfloat16).to(dev)
    WoT = torch.from_numpy(gen.bf16_normal(w.seed, "wo", (Hq * 128, w.d), (Hq * 128) ** -0.5).view(np.int16)).view(
        torch.bfloat16).to(dev)
    idx = pos_d.view(w.B, L)
    aws = cer.workspace(cer.load().cer_routed_attention_workspace_size(w.B, L, w.d, Hq, Hkv), dev)
    t_layer = device_time(torch, stream, flush, lambda: cer.cer_routed_attention(
        h, idx, WqkvT, WoT, Hq, Hkv, causal, out=hout, ws=aws, stream=stream), reps)
    cer.cer_sync_status(stream)
    proj_flops = 2.0 * w.B * L * w.d * (width + Hq * 128)
    flops = w.attn_flops(bool(causal))
    tf = flops / (t_attn * 1e-3) / 1e12
    rope_bytes = 2.0 * w.B * L * (Hq + Hkv) * 128 * 2 + 4 * w.B * L
    return {"heads": [Hq, Hkv], "packed_len": L, "causal": bool(causal),
            "rope_us": t_rope * 1e3, "rope_gbs": rope_bytes / (t_rope * 1e-3) / 1e9,
            "attention_us": t_attn * 1e3, "attention_flops": flops, "attention_tflops": tf,
            "attention_frac": tf / peak_tf, "peak_source": "bf16_tflops (burst) of measured",
            "sublayer_us": t_layer * 1e3, "sublayer_tflops": (proj_flops + flops) / (t_layer * 1e-3) / 1e12,
            "sublayer": "gather, QKV projection, rotary embedding, attention, output projection + scatter-add "
                        "(out of place)"}


def measure_ucs(cer, torch, w, h0, h, flush, stream, dev, core, exp, t, Wg, Wu, WdT, ws, inp, reps=20):
    """Time the UCS kernels on the workload's own tensors: the keep masks of two
    block calls (t and t_ref = the same inputs with t + 0.05), the redundancy
    gap of the block's input and output, and the whole block with the FFN gate
    (gate/up over all I channels, leakage of the mask's pruned channels,
    delta_FFN = 0.150 as in App. A.4)."""
    masks = []
    for dt in (0.0, 0.05):
        h.copy_(h0)
        m = torch.empty((w.B, w.N), dtype=torch.uint8, device=dev)
        cer.cer_routed_block(h, core, exp, (t + dt).clamp(max=1.0), w.task, w.r0, w.r1, w.K, Wg, Wu, WdT, None,
                             mask=m, ws=ws, stream=stream)
        masks.append(m)
    jac = torch.empty(w.B, dtype=torch.float32, device=dev)
    rda = torch.empty_like(jac)
    gap = torch.empty_like(jac)
    skip = torch.empty(w.B, dtype=torch.uint8, device=dev)
    gws = cer.workspace(cer.load().cer_redundancy_gap_workspace_size(w.B, w.N), dev)

    t_drop = device_time(torch, stream, flush, lambda: cer.cer_drop_set_stats(masks[0], masks[1], w.r0, w.r1, jac,
                                                                               None, rda, stream=stream), reps)
    t_gap = device_time(torch, stream, flush, lambda: cer.cer_redundancy_gap(h0, h, masks[1], 0.004, gap, skip,
                                                                              ws=gws, stream=stream), reps)
    cer.cer_sync_status(stream)
    gated = {}
    if w.C < w.I and w.I % 64 == 0:
        def bf(bits):
            return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)
        Wg_g, Wu_g, WdT_g, norms, _ = cer.gate_weights(bf(inp["Wg"]), bf(inp["Wu"]), bf(inp["WdT"]),
                                                       torch.from_numpy(inp["chan"]).to(dev))
        leak = torch.empty(1, dtype=torch.float32, device=dev)
        flag = torch.empty(1, dtype=torch.uint8, device=dev)
        gws2 = cer.workspace(cer.load().cer_routed_block_gated_workspace_size(
            w.B, w.N, w.d, w.Hc, w.He if w.task else 0, w.task, w.r0, w.r1, w.K, w.I), dev)

        def gated_step():
            h.copy_(h0)
            flush.fill_(1.0)

        ms = []
        for i in range(reps + 3):
            gated_step()
            torch.cuda._sleep(200000)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            cer.cer_routed_block_gated(h, core, exp, t, w.task, w.r0, w.r1, w.K, Wg_g, Wu_g, WdT_g, w.C, norms,
                                       0.150, None, leak, flag, ws=gws2, stream=stream)
            b.record(stream)
            b.synchronize()
            if i >= 3:
                ms.append(a.elapsed_time(b))
        cer.cer_sync_status(stream)
        gated = {"gated_block_ms": float(np.mean(ms)), "gated_block_tokens_per_s": w.B * w.N / (np.mean(ms) * 1e-3),
                 "ffn_leakage": round(float(leak.item()), 5), "pruned_ffn_taken": bool(flag.item()),
                 "delta_ffn": 0.150}
    gap_bytes = 2.0 * w.B * w.N * w.d * 2 + w.B * w.N
    return {"drop_set_stats_us": t_drop * 1e3, "redundancy_gap_us": t_gap * 1e3,
            "redundancy_gap_gbs": gap_bytes / (t_gap * 1e-3) / 1e9,
            "jaccard_t_vs_t+0.05": [round(float(x), 4) for x in jac.cpu().numpy()],
            "rda_t_vs_t+0.05": [round(float(x), 4) for x in rda.cpu().numpy()],
            "redundancy_gap": [round(float(x), 6) for x in gap.cpu().numpy()], **gated}


# ------------------------------------------------------------------ CPU oracle timing

def time_oracle(w: gen.Workload, inp: dict, min_seconds: float, max_reps: int = 50):
    """The oracle as it stands on one sequence of the workload, repeated until
    min_seconds; returns (tokens/s, seconds, reps)."""
    from oracle import cer_oracle as ora
    b = 0
    sl = slice(b, b + 1)
    args = (inp["h"][sl], inp["W1"], inp["w2"], inp.get("b1"), inp["t"][sl], w.task, w.r0, w.r1, w.K,
            inp["Wg"], inp["Wu"], inp["WdT"], inp["chan"], inp.get("W1e"), inp.get("w2e"), inp.get("Ue"),
            inp.get("b1e"))
    t0 = time.perf_counter()
    reps = 0
    while True:
        ora.routed_block(*args)
        reps += 1
        el = time.perf_counter() - t0
        if el >= min_seconds or reps >= max_reps:
            break
    return w.N * reps / el, el, reps


def blas_threads() -> int:
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        v = os.environ.get(var)
        if v and v.isdigit():
            return int(v)
    return os.cpu_count() or 1


def run_reference(args, info):
    """--impl reference: the CPU oracle, timed on the host cores, same workload."""
    if not info.is_root:
        return 0
    w = gen.WORKLOADS[args.config]()
    inp = gen.make_inputs(w)
    for _ in range(args.warmup):
        time_oracle(w, inp, 0.0, max_reps=1)
    times = []
    for _ in range(args.steps):
        _, el, _ = time_oracle(w, inp, 0.0, max_reps=1)
        times.append(el)
    t = float(np.mean(times))
    value = w.N / t
    sample = f"one sequence ({w.N} tokens) of {w.name} per step, full routed block in fp64 numpy"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, False),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ GPU arm

def _bf(torch, dev, bits):
    import numpy as _np
    return torch.from_numpy(_np.ascontiguousarray(bits).view(_np.int16)).view(torch.bfloat16).to(dev)


def _f32(torch, dev, a):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)


class BlockSetup:
    """One workload's tensors on the device: scorers, h (and a pristine copy,
    restored before every step since the block updates h in place), t, the FFN
    weights as kept-channel slices packed once (the static mask of App. A.4, as
    at model load) and the block's workspace."""

    def __init__(self, torch, cer, w, inp, dev, full_ffn=None):
        self.w = w
        bf = lambda bits: _bf(torch, dev, bits)  # noqa: E731
        f32 = lambda a: _f32(torch, dev, a)       # noqa: E731
        self.core = cer.Scorer(W1=bf(inp["W1"]), w2=f32(inp["w2"]), b1=f32(inp.get("b1")))
        self.exp = None
        if w.task == 1:
            self.exp = cer.Scorer(W1=bf(inp["W1e"]), w2=f32(inp["w2e"]),
                                  U=bf(inp["Ue"]) if inp.get("Ue") is not None else None)
        self.h = bf(inp["h"])
        self.h0 = self.h.clone()
        self.t = f32(inp["t"])
        Wg, Wu, WdT = full_ffn if full_ffn is not None else (bf(inp["Wg"]), bf(inp["Wu"]), bf(inp["WdT"]))
        self.pack_ms = None
        if w.C < w.I:
            chan = torch.from_numpy(inp["chan"]).to(dev)
            cer.pack_ffn_weights(Wg, Wu, WdT, chan)            # warm
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            Wg, Wu, WdT = cer.pack_ffn_weights(Wg, Wu, WdT, chan)
            e1.record()
            torch.cuda.synchronize(dev)
            self.pack_ms = e0.elapsed_time(e1)
        self.Wg, self.Wu, self.WdT = Wg, Wu, WdT
        self.ws = cer.workspace(cer.cer_routed_block_workspace_size(w.B, w.N, w.d, w.Hc, w.He if w.task else 0,
                                                                    w.task, w.r0, w.r1, w.K, w.C, False), dev)

    def step(self, cer, stream, stage_events=None):
        w = self.w
        cer.cer_routed_block(self.h, self.core, self.exp, self.t, w.task, w.r0, w.r1, w.K, self.Wg, self.Wu,
                             self.WdT, None, ws=self.ws, stage_events=stage_events, stream=stream)


def prepare_step(torch, setup, flush, i):
    """Outside the timed interval: restore h (the block updates it in place),
    evict L2 with a 256 MiB write so the step reads its inputs from HBM, and
    keep the GPU busy (a short spin) while the host enqueues the step, so host
    launch latency is not counted as device time."""
    setup.h.copy_(setup.h0)
    flush.fill_(float(i))
    torch.cuda._sleep(200000)


def time_block(torch, cer, setup, flush, stream, steps, warmup, n_stage, clocks=None, dist=None, dev=None):
    """W warm-up steps, then K steps each bracketed by CUDA events on the
    launching stream (no event between the kernels, so programmatic dependent
    launch overlaps them as in production); then a separate pass of n_stage
    steps with the library's stage events between kernels (serialised) for
    the per-stage times.  Returns (per-step ms, per-stage mean ms [5])."""
    for i in range(warmup):
        prepare_step(torch, setup, flush, i)
        setup.step(cer, stream)
    cer.cer_sync_status(stream)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    if clocks is not None:
        clocks.start()
        time.sleep(0.3)
    runtime.barrier(dist)
    torch.cuda.synchronize(dev)
    for i in range(steps):
        prepare_step(torch, setup, flush, i)
        ev[i][0].record(stream)
        setup.step(cer, stream)
        ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    runtime.barrier(dist)
    if clocks is not None:
        clocks.stop()
    cer.cer_sync_status(stream)
    step_ms = np.array([a.elapsed_time(b) for a, b in ev])
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(n_stage)]
    for i in range(n_stage):
        prepare_step(torch, setup, flush, i)
        setup.step(cer, stream, evs[i])
    torch.cuda.synchronize(dev)
    cer.cer_sync_status(stream)
    stage = np.array([[e[j].elapsed_time(e[j + 1]) for j in range(5)] for e in evs]).mean(axis=0)
    return step_ms, stage


STAGES = ("score", "topk", "gather", "ffn_gateup", "ffn_down_scatter")


def stage_report(w: gen.Workload, stage_ms, peaks) -> dict:
    """Each serialised stage against its own roofline: the algorithmic bytes
    and flops of the stage (not what the kernels happen to move), the time
    they need at the measured HBM bandwidth and at the bf16 burst peak, the
    larger of the two as the bound, and bound / measured as the fraction."""
    bw = float(peaks["hbm_gbs"]) * 1e9
    pk = float(peaks["bf16_tflops"]) * 1e12
    Ht = w.Hc + (w.He if w.task == 1 else 0)
    M, d, C, BN = w.M, w.d, w.C, w.B * w.N
    work = {
        # reads h once (+ the scorer weights); 2 B N d Ht flop
        "score": (2.0 * BN * d + 2.0 * Ht * d, 2.0 * BN * d * Ht),
        # reads the logits, writes the keep list
        "topk": (4.0 * BN + 4.0 * M, 0.0),
        # kept rows in and out, plus the keep list
        "gather": (4.0 * M * d + 4.0 * M, 0.0),
        # packed rows, gate and up slices in; act out
        "ffn_gateup": (2.0 * M * d + 4.0 * C * d + 2.0 * M * C, 4.0 * M * d * C),
        # act and down slice in; kept rows of h read and written
        "ffn_down_scatter": (2.0 * M * C + 2.0 * C * d + 4.0 * M * d, 2.0 * M * d * C),
    }
    out = {}
    for name, t_ms in zip(STAGES, stage_ms):
        nbytes, flops = work[name]
        t = float(t_ms) * 1e-3
        t_hbm, t_tc = nbytes / bw, flops / pk
        bound = "tensor" if t_tc > t_hbm else "hbm"
        r = {"us": round(t * 1e6, 2), "bound": bound, "frac": round(max(t_hbm, t_tc) / t, 4) if t > 0 else None,
             "gbs": round(nbytes / t / 1e9, 1) if t > 0 else None}
        if bound == "hbm" and t > 0:
            r["frac_vs_8tbs"] = round(nbytes / NOMINAL_HBM_BPS / t, 4)   # the nominal HBM3e figure
        if flops:
            r["tflops"] = round(flops / t / 1e12, 1) if t > 0 else None
        out[name] = r
    t_ffn = (float(stage_ms[3]) + float(stage_ms[4])) * 1e-3
    ffn_b = work["ffn_gateup"][0] + work["ffn_down_scatter"][0] - 2.0 * M * C * 2   # act stays on chip in the bound
    ffn_f = work["ffn_gateup"][1] + work["ffn_down_scatter"][1]
    out["ffn"] = {"us": round(t_ffn * 1e6, 2), "bound": "tensor" if ffn_f / pk > ffn_b / bw else "hbm",
                  "frac": round(max(ffn_f / pk, ffn_b / bw) / t_ffn, 4), "tflops": round(ffn_f / t_ffn / 1e12, 1)}
    return out


NOMINAL_HBM_BPS = 8.0e12   # GB300 HBM3e, nominal (the stages' "frac" uses the measured copy bandwidth)


def stage_floor_us(torch, cer, stream, reps=60):
    """The floor every serialised stage carries: two events on the stream with
    one near-empty library kernel between them (a bounded wait on an mbarrier
    phase that the kernel completes itself), median over `reps`."""
    ts = []
    for i in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(20000)   # keeps the host ahead, so no launch latency is timed
        a.record(stream)
        cer.cer_selftest_bounded_wait(1, arrive=True, limit_us=1000, stream=stream)
        b.record(stream)
        ts.append((a, b))
    torch.cuda.synchronize()
    cer.cer_sync_status(stream)
    return float(np.median([a.elapsed_time(b) * 1e3 for a, b in ts[reps // 6:]]))


SWEEP_N = (1024, 2048, 4096, 8192, 16384)
SWEEP_R = (0.1, 0.3, 0.5, 0.7, 0.9)
SWEEP_F = (0.25, 0.5, 1.0)


def sweep_points(torch, cer, dev, flush, stream, peaks, steps=5, warmup=3, ffn_bits=None):
    """The 7B sweep (B = 1, d = 3584, I = 18944, all routable, generation) on
    the whole grid N x token keep ratio x FFN keep ratio.  The inputs of every
    point are those of gen.sweep(N, r, f) (h, scorer weights and t depend on
    N only; the channel keep set on the FFN ratio only), so each N's tensors
    and each ratio's packed weight slices are made once.  Yields one dict per
    point: the whole step (L2 flushed between steps) and every stage against
    its roofline."""
    if ffn_bits is None:    # the FFN weights of (seed 0, I = 18944, d = 3584), drawn once
        base = gen.make_inputs(gen.sweep(SWEEP_N[0], 0.5, 1.0))
        ffn_bits = (base["Wg"], base["Wu"], base["WdT"])
    full = tuple(_bf(torch, dev, x) for x in ffn_bits)
    packed = {}
    for f in SWEEP_F:
        w = gen.sweep(SWEEP_N[0], 0.5, f)
        if w.C < w.I:
            chan = torch.from_numpy(gen.channel_keep_set(w.seed, "chan", w.I, w.C)).to(dev)
            packed[f] = cer.pack_ffn_weights(*full, chan)
        else:
            packed[f] = full
    for n in SWEEP_N:
        inp = gen.make_inputs(gen.sweep(n, 0.5, 1.0), ffn_weights=ffn_bits)
        setup = BlockSetup(torch, cer, gen.sweep(n, 0.5, 1.0), inp, dev, full_ffn=full)
        for r in SWEEP_R:
            for f in SWEEP_F:
                w = gen.sweep(n, r, f)
                setup.w = w
                setup.Wg, setup.Wu, setup.WdT = packed[f]
                setup.ws = cer.workspace(cer.cer_routed_block_workspace_size(w.B, w.N, w.d, w.Hc, w.He, w.task,
                                                                             w.r0, w.r1, w.K, w.C, False), dev)
                step_ms, stage = time_block(torch, cer, setup, flush, stream, steps, warmup, steps, dev=dev)
                ms = float(step_ms.mean())
                yield {"N": n, "token_ratio": r, "ffn_ratio": f, "K": w.K, "M": w.M, "C": w.C,
                       "ms_per_step": round(ms, 4), "tokens_per_s": w.B * w.N / (ms * 1e-3),
                       "stages": stage_report(w, stage, peaks)}
        del setup
    del full, packed


def sweep_summary(points) -> dict:
    """min / median / max over the sweep's points of every stage's roofline
    fraction (and of the whole step's tokens/s)."""
    out = {"points": len(points),
           "grid": {"N": list(SWEEP_N), "token_ratio": list(SWEEP_R), "ffn_ratio": list(SWEEP_F)}}
    for name in STAGES + ("ffn",):
        fr = np.array([p["stages"][name]["frac"] for p in points], dtype=np.float64)
        out[f"{name}_frac"] = {"min": round(float(fr.min()), 4), "median": round(float(np.median(fr)), 4),
                               "max": round(float(fr.max()), 4)}
    tps = np.array([p["tokens_per_s"] for p in points])
    out["tokens_per_s"] = {"min": float(tps.min()), "median": float(np.median(tps)), "max": float(tps.max())}
    out["per_point"] = [[p["N"], p["token_ratio"], p["ffn_ratio"], p["ms_per_step"],
                         [p["stages"][k]["us"] for k in STAGES], [p["stages"][k]["frac"] for k in STAGES],
                         p["stages"]["ffn"]["frac"]] for p in points]
    out["per_point_fields"] = ["N", "token_ratio", "ffn_ratio", "ms_per_step", "stage_us (" + ", ".join(STAGES) + ")",
                               "stage_frac", "ffn_frac"]
    return out


def run_gpu(args, info):
    import torch
    from paper_2608_29291_gb300 import cer

    torch.cuda.set_device(info.local_rank)
    dev = torch.device("cuda", info.local_rank)
    dist = runtime.init_group(info, "nccl")
    cer.load()
    peaks, peak_kind = load_peaks()
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    base = gen.WORKLOADS[args.config]()
    w = gen.Workload(**{**base.__dict__, "seed": runtime.replica_seed(base.seed, info.rank)})
    inp = gen.make_inputs(w)
    S = BlockSetup(torch, cer, w, inp, dev)
    core, exp, h, h0, t = S.core, S.exp, S.h, S.h0, S.t
    Wg, Wu, WdT, ws = S.Wg, S.Wu, S.WdT, S.ws
    chan = None

    # ---- device-timed region: K steps, L2 flushed between steps
    clocks = ClockSampler(smi_index(info.local_rank))
    n_stage = max(3, min(args.steps, 50))
    step_ms, stage = time_block(torch, cer, S, flush, stream, args.steps, args.warmup, n_stage, clocks=clocks,
                                dist=dist, dev=dev)
    mean_ms = float(step_ms.mean())
    slow_ms = runtime.max_over_ranks(dist, mean_ms, device=dev)
    tokens = w.B * w.N * info.world
    value = tokens / (slow_ms * 1e-3)
    floor_us = round(stage_floor_us(torch, cer, stream), 2)

    # ---- end to end through the public API: pinned host h in, h out.  Every
    # step uploads its own h (and t) from pinned host memory, runs the block,
    # and downloads its output.  Three streams and four device buffers overlap
    # the uploads and downloads of neighbouring steps with the compute, as a
    # serving loop would (with two buffers a buffer's upload, compute and
    # download run back to back every two steps, which the host link -- about
    # 190 GB/s each way, 315 GB/s both ways together on GB300 -- cannot hide).
    # Instead of an L2 flush inside the timed loop, consecutive steps take
    # different copies of the scorer and FFN weights (as the layers of a model
    # would), so many that the copies a step does not use exceed the flush
    # size: every step reads its weights from HBM.  The serialised time of one
    # step (upload, compute, download back to back) is reported beside it.
    set_bytes = sum(x.numel() * x.element_size() for x in (Wg, Wu, WdT))
    n_sets = 1 + -(-FLUSH_BYTES // set_bytes)

    def clone_scorer(sc):
        if sc is None:
            return None
        return cer.Scorer(W1=sc.W1.clone(), w2=sc.w2.clone(), b1=None if sc.b1 is None else sc.b1.clone(),
                          U=None if sc.U is None else sc.U.clone())

    layers = [(core, exp, Wg, Wu, WdT)] + [(clone_scorer(core), clone_scorer(exp), Wg.clone(), Wu.clone(), WdT.clone())
                                           for _ in range(n_sets - 1)]
    h_host = torch.from_numpy(np.ascontiguousarray(inp["h"]).view(np.int16)).view(torch.bfloat16).pin_memory()
    t_host = torch.from_numpy(np.ascontiguousarray(inp["t"], dtype=np.float32)).pin_memory()
    nbuf = 4
    h_buf = [torch.empty_like(h) for _ in range(nbuf)]
    t_buf = [torch.empty_like(t) for _ in range(nbuf)]
    out_host = [torch.empty_like(h_host).pin_memory() for _ in range(nbuf)]
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(nbuf)]
    ev_cmp = [torch.cuda.Event() for _ in range(nbuf)]
    ev_out = [torch.cuda.Event() for _ in range(nbuf)]
    e2e_steps = max(3, min(args.steps, 50))

    def e2e_step(i, serial=False):
        k = i % nbuf
        if i >= nbuf:
            s_in.wait_event(ev_out[k])           # this buffer's previous download is done
        with torch.cuda.stream(s_in):
            h_buf[k].copy_(h_host, non_blocking=True)
            t_buf[k].copy_(t_host, non_blocking=True)
            ev_in[k].record(s_in)
        stream.wait_event(ev_in[k])
        l_core, l_exp, l_wg, l_wu, l_wdt = layers[i % n_sets]
        cer.cer_routed_block(h_buf[k], l_core, l_exp, t_buf[k], w.task, w.r0, w.r1, w.K, l_wg, l_wu, l_wdt, chan,
                             ws=ws, stream=stream)
        ev_cmp[k].record(stream)
        s_out.wait_event(ev_cmp[k])
        with torch.cuda.stream(s_out):
            out_host[k].copy_(h_buf[k], non_blocking=True)
            ev_out[k].record(s_out)
        if serial:
            s_in.wait_event(ev_out[k])
            stream.wait_event(ev_out[k])

    for i in range(3):
        e2e_step(i)
    torch.cuda.synchronize(dev)
    runtime.barrier(dist)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    stream.wait_event(e0)
    for i in range(e2e_steps):
        e2e_step(i)
    e1.record(s_out)
    torch.cuda.synchronize(dev)
    e2e_ms = runtime.max_over_ranks(dist, e0.elapsed_time(e1) / e2e_steps, device=dev)
    # one step at a time: upload, compute and download back to back
    e0.record(s_in)
    stream.wait_event(e0)
    for i in range(e2e_steps):
        e2e_step(i, serial=True)
    e1.record(s_out)
    torch.cuda.synchronize(dev)
    cer.cer_sync_status(stream)
    serial_ms = runtime.max_over_ranks(dist, e0.elapsed_time(e1) / e2e_steps, device=dev)
    if not torch.equal(out_host[(e2e_steps - 1) % nbuf], out_host[(e2e_steps - 2) % nbuf]):
        raise RuntimeError("end-to-end steps on the same input disagree")
    h2d = h_host.numel() * 2 + t_host.numel() * 4
    d2h = out_host[0].numel() * 2
    del layers, h_buf, out_host

    # ---- UCS statistics on this step's tensors (Sec. 3.4): drop-set J/RDA of
    # two keep masks, redundancy gap of the block's input and output
    ucs = measure_ucs(cer, torch, w, h0, h, flush, stream, dev, core, exp, t, Wg, Wu, WdT, ws, inp)
    # ---- attention on the packed sequence (Sec. 3.4): rotary embedding and
    # softmax attention over the retained tokens, with the backbone's heads
    attn = measure_attention(cer, torch, w, flush, stream, dev, float(peaks["bf16_tflops"]))
    pack_ms = S.pack_ms
    del S

    # ---- the other full-size configs (each its own step, stages and
    # roofline fractions) and the whole 7B sweep grid, on rank 0 only
    others, sweep = {}, None
    if info.is_root and not args.quick:
        for name in ("und_1p5b", "gen_1p5b", "long_7b"):
            if name == args.config:
                continue
            wo = gen.WORKLOADS[name]()
            so = BlockSetup(torch, cer, wo, gen.make_inputs(wo), dev)
            sm, st = time_block(torch, cer, so, flush, stream, max(5, min(args.steps, 20)), 3,
                                max(5, min(args.steps, 20)), dev=dev)
            others[name] = {"workload": wo.name, "B": wo.B, "N": wo.N, "d": wo.d, "kept_rows": wo.M,
                            "kept_channels": wo.C, "ms_per_step": float(sm.mean()),
                            "tokens_per_s": wo.B * wo.N / (float(sm.mean()) * 1e-3),
                            "stages": stage_report(wo, st, peaks)}
            del so
        s7 = gen.sweep(SWEEP_N[0], 0.5, 1.0)
        same = (w.seed, w.I, w.d) == (s7.seed, s7.I, s7.d)
        sweep = sweep_summary(list(sweep_points(torch, cer, dev, flush, stream, peaks,
                                                ffn_bits=(inp["Wg"], inp["Wu"], inp["WdT"]) if same else None)))

    if not info.is_root:
        return 0

    score_ms, topk_ms, gather_ms, gateup_ms, down_ms = (float(x) for x in stage)
    gateup_flops = 4.0 * w.M * w.d * w.C
    achieved = gateup_flops / (gateup_ms * 1e-3) / 1e12
    peak = float(peaks["bf16_tflops"])
    down_flops = 2.0 * w.M * w.d * w.C
    gather_bytes = 4.0 * w.M * w.d + 4.0 * w.M

    cpu = None
    if info.world == 1 and not args.no_cpu_baseline:
        cps, el, reps = time_oracle(w, inp, args.cpu_seconds)
        cpu = {"value": cps, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
               "sample": f"{reps} x one sequence ({w.N} tokens) of {w.name}, full routed block, fp64 numpy, "
                         f"{el:.1f} s"}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": info.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": slow_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(w, True),
        "roofline": {"kernel": "ffn gate/up GEMM (tcgen05 pair MMA, SwiGLU epilogue)", "bound": "tensor",
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                     "peak_source": f"bf16_tflops (burst) of {peak_kind}",
                     "algorithmic_flops_per_launch": gateup_flops,
                     "traffic": profiled_traffic(w.name)},
        "stages_ms": {"score": score_ms, "topk": topk_ms, "gather": gather_ms, "ffn_gateup": gateup_ms,
                      "ffn_down_scatter": down_ms},
        "stages": stage_report(w, stage, peaks),
        "gather_gbs": gather_bytes / (gather_ms * 1e-3) / 1e9,
        "ffn_weights": "kept-channel slices packed once from the full weights by cer_pack_ffn_weights "
                       f"(static mask; {pack_ms:.3f} ms, not part of a step)" if pack_ms is not None else
                       "all channels",
        "ffn_tflops": (gateup_flops + down_flops) / ((gateup_ms + down_ms) * 1e-3) / 1e12,
        "score_tflops": w.score_flops() / (score_ms * 1e-3) / 1e12,
        "cpu_baseline": cpu,
        "e2e": {"value": tokens / (e2e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                "pipelining": "uploads and downloads of neighbouring steps overlap step i's compute on "
                              "separate streams (four device buffers)",
                "l2": f"not flushed: steps cycle through {n_sets} copies of the scorer and FFN weights "
                      f"({n_sets * set_bytes / 2**20:.0f} MiB of FFN weights, the unused copies > the 256 MiB "
                      f"flush), so every step reads its weights from HBM",
                "serial_ms_per_step": serial_ms,
                "serial_value": tokens / (serial_ms * 1e-3)},
        "ucs": {**ucs, "redundancy_gap_hbm_frac": ucs["redundancy_gap_gbs"] / float(peaks["hbm_gbs"]),
                "peak_source": f"hbm_gbs of {peak_kind}"},
        "attention": {**attn, "rope_hbm_frac": attn["rope_gbs"] / float(peaks["hbm_gbs"])},
        "other_configs": others or None,
        "sweep_7b": sweep,
        "stage_peaks": f"hbm_gbs and bf16_tflops (burst) of {peak_kind}",
        "gpu_launches": kernels_per_step(w.task) * args.steps,
        "stage_pass": f"per-stage times from a separate pass of {n_stage} steps with events between kernels",
        "stage_floor_us": {"value": floor_us,
                           "what": "median time between two events with one near-empty library kernel between "
                                   "them: the event and launch cost each serialised stage carries on top of its "
                                   "kernels (the overlapped step does not pay it)"},
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_sweep(args):
    """The 7B sweep on the whole grid, one JSON line per point."""
    import torch
    from paper_2608_29291_gb300 import cer

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    cer.load()
    peaks, peak_kind = load_peaks()
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    for p in sweep_points(torch, cer, dev, flush, stream, peaks, steps=args.steps, warmup=args.warmup):
        p["peak_source"] = f"hbm_gbs / bf16_tflops (burst) of {peak_kind}"
        p["l2"] = "flushed between timed steps"
        print(json.dumps(p), flush=True)
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("cer", "reference"), default="cer")
    ap.add_argument("--config", choices=sorted(gen.WORKLOADS), default="long_7b")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--quick", action="store_true",
                    help="leave out the other configs and the sweep (the headline workload's line only)")
    ap.add_argument("--sweep", action="store_true",
                    help="time the 7B sweep grid (one JSON line per point) instead of the bench line")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    info = runtime.rank_info()
    if args.sweep:
        return run_sweep(args)
    if args.impl == "reference":
        return run_reference(args, info)
    return run_gpu(args, info)


if __name__ == "__main__":
    sys.exit(main())
