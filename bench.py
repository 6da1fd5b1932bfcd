#!/usr/bin/env python3
"""Benchmark of the low-bit MLA decode hot path on GB300.

One step = qmla_quant_append of one new token per sequence followed by
qmla_mla_decode over every cached token (plan, main and merge kernels), on
the DeepSeek-V3-shaped workload (64 sequences x 128 heads, 4096 cached tokens
plus the appended one, INT4 content + INT4 RoPE key) unless --workload says
otherwise. The metric is KV-tokens/s: tokens attended per step / step time.
The default run then measures the other workloads the same way and reports
them under "configs" (the 128-sequence serving mix over its 256 steps, also on
the BF16 comparison cache, and the DeepSeek-V3 workload on the BF16 cache).

Contract: `python bench.py --gpus N --steps K --warmup W` prints one JSON line
(rank 0). With N > 1 (torchrun) every rank decodes its own copy of the
workload (independent sequences, no collective on the data path): weak
scaling, max time over ranks. `--impl reference` times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from workloads import synthetic as W  # noqa: E402

METRIC = "low-bit MLA decode KV-tokens/s and µs/step on 1 GB300; % of roofline"
UNIT = "KV-tokens/s"
DEFAULT_WORKLOAD = "dsv3_b64_h128_l4096_int4"
TAU = 1.0 / math.sqrt(192.0)
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(W.WORKLOADS))
    ap.add_argument("--bf16-cache", action="store_true", help="decode the BF16 comparison cache instead")
    ap.add_argument("--protect", action="store_true",
                    help="sink4/local128 BF16 protection (the paper's C4R4 serving configuration)")
    ap.add_argument("--c4r4", action="store_true",
                    help="store the INT4 cache in the paper's own 20,480-byte page (bf16/fp32 scales, uint8 zeros)")
    ap.add_argument("--q-tokens", type=int, default=1,
                    help="query tokens per sequence (multi-token prediction / speculative verification); each step "
                         "appends that many tokens and scores them under the causal mask")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other workloads (configs) measured after the headline one")
    ap.add_argument("--trace", default=None, metavar="NPZ",
                    help="instead of timing: build the trace library, trace one decode step's main kernel, print "
                         "the per-tile stage breakdown and save the raw clock64 stamps to NPZ")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args(argv)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x: float, dist, device) -> float:
    """The largest x over all ranks (x itself without a process group): the job's
    time is its slowest rank's."""
    if dist is None:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(world: int, tokens_per_rank_step: float, ms_per_step: float) -> float:
    """KV tokens per second over all ranks: every rank decodes its own replica of
    the workload in the same (slowest-rank) step time."""
    return world * tokens_per_rank_step / (ms_per_step * 1e-3)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"])}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def workload_cost(w: W.Workload, lens: list[int], bf16: bool, c4r4: bool = False, q_tokens: int = 1):
    """Algorithmic FLOPs and HBM bytes of one decode launch (see the design notes).
    With T query tokens per sequence every cached token is scored by T x H query
    rows (the causal mask hides T(T-1)/2 of a sequence's pairs; not subtracted)."""
    tokens = sum(lens)
    rows = q_tokens * w.heads
    flops = 2.0 * rows * (576 + 512) * tokens
    per_tok = 1152 if bf16 else (320 if c4r4 else (324 if w.c_bits == 4 else 196))
    nbytes = tokens * per_tok + w.batch * rows * (576 * 2 + 512 * 4 + 4)
    return flops, nbytes


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled while the timed loop runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.12)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"], f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def profile_traffic(kernel_file_hash: str, workload: str, bf16: bool = False, protect: bool = False,
                    c4r4: bool = False, q_tokens: int = 1):
    """The committed ncu record of DRAM bytes per main-kernel launch for this
    workload and cache variant, if it was taken on the current kernel sources;
    otherwise None."""
    p = os.path.join(ROOT, "profiles", "decode_main_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    if d.get("decode_cu_sha256") != kernel_file_hash:
        return None
    for r in d.get("records", []):
        if (r.get("workload") == workload and bool(r.get("bf16_cache")) == bool(bf16)
                and bool(r.get("protect")) == bool(protect) and bool(r.get("c4r4")) == bool(c4r4)
                and int(r.get("q_tokens", 1)) == q_tokens):
            return r
    return None


# The sources decode_main is compiled from (its translation unit and headers).
DECODE_MAIN_SOURCES = ("common.cuh", "decode.cu", "kernels.h", "ptx.cuh")


def decode_cu_hash() -> str:
    """sha256 over the sources decode_main is compiled from (and the public
    header they include), so a traffic figure taken on another version of the
    kernel is not used."""
    d = os.path.join(ROOT, "paper_2609_36760_gb300", "csrc")
    h = hashlib.sha256()
    paths = [os.path.join(d, n) for n in DECODE_MAIN_SOURCES] + [os.path.join(ROOT, "include", "qmla.h")]
    for path in paths:
        with open(path, "rb") as f:
            h.update(os.path.basename(path).encode() + b"\0" + f.read())
    return h.hexdigest()


# ------------------------------------------------------------------ native
class Workspace:
    """GPU state of one workload: pool, block table, per-step inputs."""

    def __init__(self, w: W.Workload, bf16: bool, dev: torch.device, nsteps: int, protect: bool = False,
                 c4r4: bool = False, q_tokens: int = 1, gen_device=None):
        """gen_device None draws the inputs with the host generators (the values the
        oracle sees); a CUDA device draws them there (same distributions)."""
        import paper_2609_36760_gb300 as Q
        self.Q = Q
        self.q_tokens = q_tokens
        if q_tokens > 1:
            if bf16 or c4r4:
                raise SystemExit("--q-tokens > 1 runs on the INT4/INT2 block (protection optional)")
            w = dataclasses.replace(w, append=max(w.append, q_tokens))  # the scored tokens are the appended ones
        self.w, self.bf16, self.dev = w, bf16, dev
        self.protect = protect and not bf16
        self.c4r4 = c4r4 and not bf16
        if self.c4r4 and w.c_bits != 4:
            raise SystemExit("--c4r4 stores INT4 content: pick a workload with c_bits = 4")
        self.prefill = W.seq_lengths(w)
        table, nblocks = W.block_table(w)
        self.table = table.to(dev)
        bb = Q.bf16_block_bytes() if bf16 else (Q.c4r4_page_bytes() if self.c4r4 else Q.block_bytes(w.c_bits))
        self.pool = torch.zeros((nblocks, bb), dtype=torch.uint8, device=dev)
        self.err = torch.zeros(1, dtype=torch.int32, device=dev)
        # per-request 132 x 576 bf16 protection rows (152,064 bytes each)
        self.prot = (torch.zeros((w.batch, 132, 576), dtype=torch.bfloat16, device=dev) if self.protect else None)
        self.prefill_lens = torch.tensor(self.prefill, dtype=torch.int32, device=dev)
        gains = W.channel_gains(w)
        self.nsteps = max(1, min(nsteps, w.steps))
        self.step_in = [dict(lat=[], kp=[], pos=[]) for _ in range(self.nsteps)]
        # Prefill through the library, one sequence at a time (bounded host memory).
        for b in range(w.batch):
            n_all = self.prefill[b] + w.append * self.nsteps
            lat = W.latent_for_seq(w, b, n_all, gains, device=gen_device)
            kp = W.kpe_for_seq(w, b, n_all, device=gen_device)
            n = self.prefill[b]
            self._append(lat[:n].to(dev), kp[:n].to(dev), torch.full((n,), b, dtype=torch.int32, device=dev),
                         torch.arange(n, dtype=torch.int32, device=dev), self.prefill_lens)
            for s in range(self.nsteps):
                for k in range(w.append):
                    p = n + w.append * s + k
                    self.step_in[s]["lat"].append(lat[p:p + 1])
                    self.step_in[s]["kp"].append(kp[p:p + 1])
                    self.step_in[s]["pos"].append(p)
        torch.cuda.synchronize(dev)
        self.steps = []
        for s in range(self.nsteps):
            si = self.step_in[s]
            ql, qp = W.queries(w, s, device=gen_device) if q_tokens == 1 else W.queries_multi(w, s, q_tokens)
            lens = [n + w.append * (s + 1) for n in self.prefill]
            host = {
                "lat": torch.cat(si["lat"]) if si["lat"] else torch.zeros(0, 512, dtype=torch.bfloat16),
                "kp": torch.cat(si["kp"]) if si["kp"] else torch.zeros(0, 64, dtype=torch.bfloat16),
                "sid": torch.tensor([b for b in range(w.batch) for _ in range(w.append)], dtype=torch.int32),
                "pos": torch.tensor(si["pos"], dtype=torch.int32),
                "ql": ql.contiguous(), "qp": qp.contiguous(),
                "lens": torch.tensor(lens, dtype=torch.int32),
            }
            if gen_device is not None:
                host = {k: v.cpu() for k, v in host.items()}
            self.steps.append({"host": host, "dev": {k: v.to(dev) for k, v in host.items()}, "lens": lens})
        qshape = (w.batch, w.heads) if q_tokens == 1 else (w.batch, q_tokens, w.heads)
        self.out = torch.empty(qshape + (512,), dtype=torch.float32, device=dev)
        self.lse = torch.empty(qshape, dtype=torch.float32, device=dev)
        self.ws = Q.workspace_for(w.batch, q_tokens * w.heads, dev)

    def _append(self, lat, kp, sid, pos, lens_after=None):
        if lat.shape[0] == 0:
            return
        if self.c4r4:
            self.Q.quant_append_c4r4(self.pool, lat, kp, sid, pos, self.table, self.err,
                                     seq_lens=lens_after if self.protect else None, prot=self.prot)
        elif self.protect:
            self.Q.quant_append_protected(self.pool, self.w.c_bits, lat, kp, sid, pos, self.table, lens_after,
                                          self.prot, self.err)
        elif self.bf16:
            self.Q.bf16_append(self.pool, lat, kp, sid, pos, self.table, self.err)
        else:
            self.Q.quant_append(self.pool, self.w.c_bits, lat, kp, sid, pos, self.table, self.err)

    def step(self, s: int, d: dict | None = None, out=None, lse=None):
        d = d if d is not None else self.steps[s % self.nsteps]["dev"]
        out = self.out if out is None else out
        lse = self.lse if lse is None else lse
        self._append(d["lat"], d["kp"], d["sid"], d["pos"], d["lens"])
        self.decode(d, out, lse)

    def cache_kind(self):
        return "bf16" if self.bf16 else ("c4r4" if self.c4r4 else self.w.c_bits)

    def decode(self, d: dict, out, lse, events=None):
        """One decode call through the variant's own entry point; with events
        (before, after) through qmla_mla_decode_ex, which records them around the
        main kernel of this call."""
        if events is not None:
            self.Q.mla_decode_ex(self.pool, self.cache_kind(), d["ql"], d["qp"], self.table, d["lens"], TAU, out,
                                 lse, self.ws, self.err, prot=self.prot, events=events)
        elif self.q_tokens > 1:
            self.Q.mla_decode_multi(self.pool, self.w.c_bits, d["ql"], d["qp"], self.table, d["lens"], TAU, out,
                                    lse, self.ws, self.err, prot=self.prot)
        elif self.c4r4:
            self.Q.mla_decode_c4r4(self.pool, d["ql"], d["qp"], self.table, d["lens"], TAU, out, lse, self.ws,
                                   self.err, prot=self.prot)
        elif self.protect:
            self.Q.mla_decode_protected(self.pool, self.w.c_bits, d["ql"], d["qp"], self.table, d["lens"], self.prot,
                                        TAU, out, lse, self.ws, self.err)
        elif self.bf16:
            self.Q.mla_decode_bf16cache(self.pool, d["ql"], d["qp"], self.table, d["lens"], TAU, out, lse, self.ws,
                                        self.err)
        else:
            self.Q.mla_decode(self.pool, self.w.c_bits, d["ql"], d["qp"], self.table, d["lens"], TAU, out, lse,
                              self.ws, self.err)

    def launches_per_step(self) -> int:
        return (1 if self.w.append > 0 else 0) + 3


def time_steps(state: Workspace, K: int, Wm: int, flush, dev, clocks=None, dist=None):
    """Warm-up, then pass A (K whole steps as a user runs them: the library's
    launches overlap their start-up; CUDA events around each step) and pass B
    (min(K, 100) steps whose main decode kernel is bracketed by per-call events,
    which make the call's launches wait for one another in full). The L2 is
    flushed (256 MB write) before every step of both passes."""
    Q = state.Q
    stream = torch.cuda.current_stream(dev)
    for i in range(Wm):
        flush.zero_()
        state.step(i)
    torch.cuda.synchronize(dev)
    if Q.read_dev_err(state.err) != 0:
        raise RuntimeError(f"device error word {Q.read_dev_err(state.err):#x} after warm-up")
    Km = min(K, 100)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    # pass B events: before the append, after it, around the main kernel (recorded by the library), after the call
    evm = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(Km)]
    for e in ev + evm:
        for x in e:
            x.record(stream)
    torch.cuda.synchronize(dev)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    if clocks is not None:
        clocks.start()
        time.sleep(0.15)
    t_wall0 = time.perf_counter()
    for i in range(K):
        e0, e1 = ev[i]
        flush.zero_()
        e0.record(stream)
        state.step(Wm + i)
        e1.record(stream)
    torch.cuda.synchronize(dev)
    t_wall = time.perf_counter() - t_wall0
    for i in range(Km):
        a0, a1, m0, m1, e_end = evm[i]
        flush.zero_()
        d = state.steps[(Wm + i) % state.nsteps]["dev"]
        a0.record(stream)
        state._append(d["lat"], d["kp"], d["sid"], d["pos"], d["lens"])  # the same appends again: cache unchanged
        a1.record(stream)
        state.decode(d, state.out, state.lse, events=(m0, m1))
        e_end.record(stream)
    torch.cuda.synchronize(dev)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    clk = clocks.stop() if clocks is not None else None
    err = Q.read_dev_err(state.err)
    if err != 0:
        raise RuntimeError(f"device error word {err:#x} in the timed loop")
    med = lambda xs: statistics.median(xs) * 1e3  # noqa: E731
    parts_us = {"append": round(med([e[0].elapsed_time(e[1]) for e in evm]), 2),
                "prep_and_gaps": round(med([e[1].elapsed_time(e[2]) for e in evm]), 2),
                "main": round(med([e[2].elapsed_time(e[3]) for e in evm]), 2),
                "merge_and_gap": round(med([e[3].elapsed_time(e[4]) for e in evm]), 2),
                "note": "medians of pass B, whose events serialise the launches"}
    step_ms = [ev[i][0].elapsed_time(ev[i][1]) for i in range(K)]
    main_ms = [evm[i][2].elapsed_time(evm[i][3]) for i in range(Km)]
    lens_all = [state.steps[(Wm + i) % state.nsteps]["lens"] for i in range(K)]
    return {"step_ms": step_ms, "main_ms": main_ms, "parts_us": parts_us, "clocks": clk, "wall_s": t_wall,
            "tokens_per_step": sum(sum(l) for l in lens_all) / K, "lens0": lens_all[0]}


def roofline(w: W.Workload, lens, bf16: bool, c4r4: bool, q_tokens: int, ms_main: float):
    """Roofline of the main decode kernel: the slower of algorithmic FLOPs over
    the measured bf16 tensor peak and algorithmic bytes over the measured HBM
    copy bandwidth; achieved = the bound's quantity / the kernel's event time."""
    peaks, peak_src = load_peaks()
    flops, nbytes = workload_cost(w, lens, bf16, c4r4, q_tokens)
    t_tc = flops / (peaks["bf16_tflops"] * 1e12)
    t_hbm = nbytes / (peaks["hbm_gbs"] * 1e9)
    if t_tc >= t_hbm:
        achieved = flops / (ms_main * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": round(achieved, 2), "peak": peaks["bf16_tflops"], "unit": "TFLOP/s"}
    else:
        achieved = nbytes / (ms_main * 1e-3) / 1e9
        roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s"}
    roof["frac"] = round(achieved / roof["peak"], 4)
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"
    roof["kernel_us"] = round(ms_main * 1e3, 2)
    roof["algorithmic_flops"] = flops
    roof["algorithmic_bytes"] = nbytes
    roof["roofline_us"] = round(max(t_tc, t_hbm) * 1e6, 2)
    return roof


def run_native(args, ws_world: int, rank: int, local: int):
    import paper_2609_36760_gb300 as Q
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    Q.lib()
    dist = None
    if ws_world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    w = W.WORKLOADS[args.workload]
    K, Wm = args.steps, args.warmup
    state = Workspace(w, args.bf16_cache, dev, K + Wm, protect=args.protect, c4r4=args.c4r4, q_tokens=args.q_tokens)
    w = state.w
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # larger than the 126 MB L2
    t = time_steps(state, K, Wm, flush, dev, clocks=ClockSampler(local), dist=dist)
    step_ms, main_ms = t["step_ms"], t["main_ms"]
    med = lambda xs: statistics.median(xs) * 1e3  # noqa: E731
    qs = statistics.quantiles(step_ms, n=10) if K >= 10 else [min(step_ms)] * 9
    step_dist_us = {"median": round(med(step_ms), 2), "p10": round(qs[0] * 1e3, 2), "p90": round(qs[-1] * 1e3, 2)}
    ms_step_max = max_over_ranks(sum(step_ms) / K, dist, dev)
    ms_main = sum(main_ms) / len(main_ms)
    tok_per_step = t["tokens_per_step"]
    value = whole_job_value(ws_world, tok_per_step, ms_step_max)

    roof = roofline(w, t["lens0"], args.bf16_cache, state.c4r4, args.q_tokens, ms_main)
    prof = profile_traffic(decode_cu_hash(), args.workload, args.bf16_cache, args.protect, state.c4r4,
                           args.q_tokens)
    roof["traffic"] = prof["dram_bytes_per_launch"] if prof else None
    if prof:
        roof["traffic_source"] = "profiles/decode_main_traffic.json: " + prof["source"]
    roof["kernel"] = "decode_main"

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(state, K=min(K, 200), flush=flush, dev=dev, tokens=tok_per_step, n_world=ws_world, dist=dist)

    res = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws_world, "steps": K, "warmup": Wm,
        "ms_per_step": round(ms_step_max, 5), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f16", "data": "synthetic (seeded generators, workloads/synthetic.py)",
        "config": {"workload": w.name, "batch_per_gpu": w.batch, "heads": w.heads, "c_bits": w.c_bits,
                   "pe_bits": 4, "cache": cache_name(w, args.bf16_cache, args.protect, state.c4r4),
                   "q_tokens_per_seq": args.q_tokens, "kernel": "one CTA per SM (qmla_mla_decode)",
                   "kv_tokens_per_step_per_gpu": tok_per_step, "l2": "flushed (256 MB write) before every timed step",
                   "parallelism": f"replicas x{ws_world} (independent sequences)"},
        "us_per_step": round(ms_step_max * 1e3, 2),
        "us_per_step_dist": step_dist_us,
        "step_parts_us": t["parts_us"],
        "roofline": roof,
        "gpu_launches": state.launches_per_step() * K,
        "clocks": t["clocks"],
        "e2e": e2e,
        "wall_s_timed_loop": round(t["wall_s"], 3),
    }
    if rank == 0 and ws_world == 1 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline(w, args.bf16_cache, budget_s=15.0, protect=args.protect,
                                           c4r4=state.c4r4, q_tokens=args.q_tokens)
    if ws_world == 1 and not args.no_configs and args.workload == DEFAULT_WORKLOAD and not (
            args.bf16_cache or args.protect or args.c4r4 or args.q_tokens != 1):
        del state
        torch.cuda.empty_cache()
        res["configs"] = run_configs(dev, flush, K)
        b16 = res["configs"].get(w.name + "_bf16cache")
        if b16 is not None:  # INT4 (this line) against the same kernel on the BF16 cache
            b16["int4_speedup_step"] = round(b16["us_per_step"] / res["us_per_step"], 3)
            b16["int4_speedup_main"] = round(b16["roofline"]["kernel_us"] / roof["kernel_us"], 3)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(res), flush=True)


# The other workloads measured after the headline one (one line per config):
# (workload, BF16 comparison cache). Their inputs are drawn on the GPU with the
# same seeded distributions (the host generators would take minutes for the
# 1M-token workloads); the headline workload keeps the host generators, whose
# values the oracle baseline uses.
CONFIGS = [("tiny_b1_h16_l256_int4", False), ("int2_b32_h128_l32768", False), ("long_b4_h64_l128k", False),
           ("serve_b128_h16_mix", False), ("serve_b128_h16_mix", True), ("dsv3_b64_h128_l4096_int4", True)]


def run_configs(dev, flush, K: int) -> dict:
    """Every other workload, each timed like the headline one (time_steps): step
    time, KV-tokens/s and the main kernel's roofline fraction. The serving mix
    runs its 256 consecutive steps (append 1 token per sequence + decode), on
    the INT4 cache and on the BF16 comparison cache; the 128K workload adds the
    physical cache bytes of a 128K-token sequence against a BF16 cache."""
    import paper_2609_36760_gb300 as Q
    out = {}
    for name, bf16 in CONFIGS:
        w = W.WORKLOADS[name]
        Kc, Wc = (w.steps, 3) if w.steps > 1 else (min(K, 20), 3)
        state = Workspace(w, bf16, dev, Kc + Wc, gen_device=dev)
        t = time_steps(state, Kc, Wc, flush, dev)
        step_ms, main_ms = t["step_ms"], t["main_ms"]
        ms_step = sum(step_ms) / len(step_ms)
        ms_main = sum(main_ms) / len(main_ms)
        roof = roofline(state.w, t["lens0"], bf16, False, 1, ms_main)
        prof = profile_traffic(decode_cu_hash(), name, bf16)
        roof["traffic"] = prof["dram_bytes_per_launch"] if prof else None
        qs = statistics.quantiles(step_ms, n=10) if len(step_ms) >= 10 else [min(step_ms)] * 9
        r = {"cache": cache_name(w, bf16, False, False), "batch": w.batch, "heads": w.heads,
             "steps": Kc, "warmup": Wc, "us_per_step": round(ms_step * 1e3, 2),
             "us_per_step_dist": {"median": round(statistics.median(step_ms) * 1e3, 2),
                                  "p10": round(qs[0] * 1e3, 2), "p90": round(qs[-1] * 1e3, 2)},
             "kv_tokens_per_s": round(t["tokens_per_step"] / (ms_step * 1e-3), 1),
             "kv_tokens_per_step": t["tokens_per_step"], "step_parts_us": t["parts_us"],
             "roofline": {k: roof[k] for k in ("bound", "achieved", "peak", "unit", "frac", "kernel_us",
                                              "roofline_us", "algorithmic_bytes", "algorithmic_flops", "traffic")},
             "hbm_gbs_of_step": round(roof["algorithmic_bytes"] / (ms_step * 1e-3) / 1e9, 1),
             "gpu_launches": state.launches_per_step() * Kc,
             "inputs": "seeded, drawn on the GPU (same distributions as workloads/synthetic.py)"}
        if name == "long_b4_h64_l128k":
            blocks = (131072 + 63) // 64
            r["physical_cache_bytes_128k"] = {
                "int4_int4_block": blocks * Q.block_bytes(4), "bf16": blocks * Q.bf16_block_bytes(),
                "ratio": round(Q.bf16_block_bytes() / Q.block_bytes(4), 3),
                "paper_ratio_context": 3.59,
                "note": "values + fp16 scales + fp16 zeros of one 131072-token sequence, no protection buffer"}
        out[name + ("_bf16cache" if bf16 else "")] = r
        del state
        torch.cuda.empty_cache()
    for base in ("serve_b128_h16_mix", "dsv3_b64_h128_l4096_int4"):
        b16 = out.get(base + "_bf16cache")
        i4 = out.get(base)
        if b16 is not None:
            if i4 is None:  # the headline workload's INT4 figures are the line's own
                continue
            b16["int4_speedup_step"] = round(b16["us_per_step"] / i4["us_per_step"], 3)
            b16["int4_speedup_main"] = round(b16["roofline"]["kernel_us"] / i4["roofline"]["kernel_us"], 3)
    return out


def cache_name(w: W.Workload, bf16: bool, protect: bool, c4r4: bool) -> str:
    if bf16:
        return "bf16"
    base = "c4r4 paper page (bf16 content / fp32 rope scales, uint8 zeros)" if c4r4 else f"int{w.c_bits}/int4 packed"
    return base + (" + sink4/local128 bf16" if protect else "")


def run_e2e(state: Workspace, K: int, flush, dev, tokens: float, n_world: int, dist):
    """Same metric through the public API with the step's inputs in pinned host
    memory: every step copies its appended tokens, queries and lengths host to
    device and reads out and lse back. The copies are pipelined as a serving loop
    would run them: step i+1's inputs go in (copy stream) and step i-1's results
    come out (read-back stream) while step i computes; events order each copy
    against the step that produces or consumes it. Timed from the first input
    copy to the last read-back."""
    stream = torch.cuda.current_stream(dev)
    h2d_s = torch.cuda.Stream(dev)
    d2h_s = torch.cuda.Stream(dev)
    hs = [{k: v.pin_memory() for k, v in state.steps[s]["host"].items()} for s in range(state.nsteps)]
    dbuf = [{k: torch.empty_like(v, device=dev) for k, v in hs[0].items()} for _ in range(2)]  # inputs of steps i % 2
    outs = [torch.empty_like(state.out) for _ in range(2)]
    lses = [torch.empty_like(state.lse) for _ in range(2)]
    out_h = [torch.empty(state.out.shape, dtype=torch.float32).pin_memory() for _ in range(2)]
    lse_h = [torch.empty(state.lse.shape, dtype=torch.float32).pin_memory() for _ in range(2)]
    h2d = sum(v.numel() * v.element_size() for v in hs[0].values())
    d2h = out_h[0].numel() * 4 + lse_h[0].numel() * 4
    n = K + 3
    ev_in = [torch.cuda.Event() for _ in range(n)]
    ev_done = [torch.cuda.Event() for _ in range(n)]
    ev_out = [torch.cuda.Event() for _ in range(n)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)

    def issue(i):
        h, d = hs[i % state.nsteps], dbuf[i % 2]
        if i >= 2:  # step i - 2 has read this input buffer
            h2d_s.wait_event(ev_done[i - 2])
        with torch.cuda.stream(h2d_s):
            for k in h:
                d[k].copy_(h[k], non_blocking=True)
        ev_in[i].record(h2d_s)

    issue(0)
    for i in range(n):
        if i + 1 == 3:
            t0.record(h2d_s)  # the timed steps start with step 3's input copy
        if i + 1 < n:
            issue(i + 1)  # the next step's inputs go in while this step computes
        d = dbuf[i % 2]
        stream.wait_event(ev_in[i])
        if i >= 2:
            stream.wait_event(ev_out[i - 2])  # results buffer i % 2 has been read back
        flush.zero_()
        state.step(i, d, out=outs[i % 2], lse=lses[i % 2])
        ev_done[i].record(stream)
        d2h_s.wait_event(ev_done[i])
        with torch.cuda.stream(d2h_s):
            out_h[i % 2].copy_(outs[i % 2], non_blocking=True)
            lse_h[i % 2].copy_(lses[i % 2], non_blocking=True)
        ev_out[i].record(d2h_s)
    t1.record(d2h_s)
    torch.cuda.synchronize(dev)
    ms = max_over_ranks(t0.elapsed_time(t1) / K, dist, dev)
    return {"value": round(whole_job_value(n_world, tokens, ms), 1), "unit": UNIT, "ms_per_step": round(ms, 5),
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": K,
            "pipelined": "step i+1's inputs in and step i-1's results out overlap step i"}


# ------------------------------------------------------------------ oracle
def oracle_step_sample(w: W.Workload, bf16: bool, budget_s: float, max_seqs: int | None = None,
                       protect: bool = False, c4r4: bool = False, q_tokens: int = 1):
    """Times the CPU oracle on one decode step (append of the step's tokens,
    read-back and dequantisation of each sequence's cache, fp64 attention) for
    as many sequences as fit in `budget_s`. Returns (tokens, seconds, nseq)."""
    import numpy as np
    from oracle import attention as OA
    from oracle import layout as OL
    from oracle import multi_query as OM
    from oracle import paper_format as OF

    if q_tokens > 1:
        w = dataclasses.replace(w, append=max(w.append, q_tokens))
    prefill = W.seq_lengths(w)
    gains = W.channel_gains(w)
    ql, qp = W.queries(w, 0) if q_tokens == 1 else W.queries_multi(w, 0, q_tokens)
    tot_tok, tot_s, nseq = 0, 0.0, 0
    limit = w.batch if max_seqs is None else min(max_seqs, w.batch)
    for b in range(limit):
        n = prefill[b]
        L = n + w.append
        lat = W.latent_for_seq(w, b, L, gains).double().numpy()
        kp = W.kpe_for_seq(w, b, L).double().numpy()
        row = np.arange((L + 63) // 64, dtype=np.int64)
        if c4r4:
            pool = np.zeros((len(row), OF.PAGE_BYTES), np.uint8)
            OF.write_tokens(pool, lat[:n], kp[:n], np.zeros(n, np.int64), np.arange(n), row[None, :])
        elif not bf16:
            pool = np.zeros((len(row), OL.block_bytes(w.c_bits)), np.uint8)
            OL.write_tokens(pool, w.c_bits, lat[:n], kp[:n], np.zeros(n, np.int64), np.arange(n), row[None, :])
        t0 = time.perf_counter()
        if bf16:
            C, K = lat, kp
        elif c4r4:
            if w.append:
                OF.write_tokens(pool, lat[n:L], kp[n:L], np.zeros(L - n, np.int64), np.arange(n, L), row[None, :])
            q, s, z = OF.read_sequence(pool, row, L)
            C, K = OF.dequantize_tokens(q, s, z)
        else:
            if w.append:
                OL.write_tokens(pool, w.c_bits, lat[n:L], kp[n:L], np.zeros(L - n, np.int64), np.arange(n, L),
                                row[None, :])
            q, s, z = OL.read_sequence(pool, w.c_bits, row, L)
            C, K = OA.dequantize_tokens(q, s, z)
        if protect and not bf16:  # sink4/local128 positions attend with their bf16 values
            from oracle import protection as OP
            P = OP.protected_positions(L)
            C, K = np.array(C), np.array(K)
            C[P], K[P] = lat[P], kp[P]
        if q_tokens == 1:
            OA.attend(ql[b].double().numpy(), qp[b].double().numpy(), C, K, TAU)
        else:
            OM.attend_multi(ql[b].double().numpy(), qp[b].double().numpy(), C, K, TAU)
        tot_s += time.perf_counter() - t0
        tot_tok += L
        nseq += 1
        if tot_s >= budget_s:
            break
    return tot_tok, tot_s, nseq


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(w: W.Workload, bf16: bool, budget_s: float, protect: bool = False, c4r4: bool = False,
                 q_tokens: int = 1):
    tok, sec, nseq = oracle_step_sample(w, bf16, budget_s, protect=protect, c4r4=c4r4, q_tokens=q_tokens)
    return {"value": round(tok / sec, 1), "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
            "sample": f"{nseq} of {w.batch} sequences of one decode step ({tok} KV tokens, "
                      f"{w.heads} heads): append + cache read-back + dequantisation + fp64 attention, "
                      f"numpy with BLAS threads = host cores; {sec:.2f} s"}


def run_reference(args, ws_world: int, rank: int):
    if rank != 0:
        return
    w = W.WORKLOADS[args.workload]
    # Each step is a bounded sample: at most 4 sequences of the step.
    steps = []
    for i in range(args.warmup + args.steps):
        tok, sec, nseq = oracle_step_sample(w, args.bf16_cache, budget_s=1e9, max_seqs=min(4, w.batch),
                                            protect=args.protect, c4r4=args.c4r4 and not args.bf16_cache,
                                            q_tokens=args.q_tokens)
        if i >= args.warmup:
            steps.append((tok, sec))
    tok = sum(t for t, _ in steps)
    sec = sum(s for _, s in steps)
    value = tok / sec
    res = {"impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws_world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * sec / len(steps), 3),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic (seeded generators, workloads/synthetic.py)",
           "config": {"workload": w.name, "batch_per_gpu": w.batch, "heads": w.heads, "c_bits": w.c_bits,
                      "pe_bits": 4, "cache": cache_name(w, args.bf16_cache, args.protect, args.c4r4),
                      "q_tokens_per_seq": args.q_tokens,
                      "sample_per_step": f"{min(4, w.batch)} sequences"},
           "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                            "sample": f"{min(4, w.batch)} of {w.batch} sequences per step, {len(steps)} steps"},
           "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(res), flush=True)


TRACE_CTAS, TRACE_EVENTS, TRACE_TILES = 8, 128, 32


def main_trace_summary(ev):
    """Median stage lengths (cycles) of decode_main's steady tiles (2 .. n-2 of
    each traced CTA). Event numbers as stamped in decode.cu: MMA issuer 0: 1
    loop top, 112 + k QK of chunk k issued, 12 its QK committed, 14 P seen, 15
    its PV issued; issuer j: 24 + j its PV block committed; worker warp 0: 0
    loop top, 105 first chunk computed, 16 scores seen, 19 P written, 17 every
    warp's P seen, 18 row sums added; lane 0 of worker warp w: 88 + w the
    previous PV's completion seen, 48 + 5 w + kc chunk step kc arrived, 32 + w
    tile dequantised and the next tile's rows fetched."""
    import numpy as np

    stages, period = {}, []
    for c in range(ev.shape[0]):
        n = int((ev[c, 12] > 0).sum())
        for it in range(2, n - 1):
            g, nx = ev[c, :, it], ev[c, :, it + 1]
            period.append(nx[14] - g[14])
            for name, v in (("issuer 0: QK chunk 0 -> chunk 8 issued", g[120] - g[112]),
                            ("issuer 0: QK chunk 8 issued -> committed", g[12] - g[120]),
                            ("issuer 0: QK committed -> P seen", g[14] - g[12]),
                            ("issuer 0: P seen -> PV issued", g[15] - g[14]),
                            ("issuer 0: PV issued -> next QK chunk 0", nx[112] - g[15]),
                            ("warp 0: QK committed -> scores seen", g[16] - g[12]),
                            ("warp 0: scores seen -> P written", g[19] - g[16]),
                            ("warp 0: P written -> all P seen", g[17] - g[19]),
                            ("warp 0: all P seen -> row sums added", g[18] - g[17]),
                            ("warp 0: row sums added -> next loop top", nx[0] - g[18]),
                            ("warp 0: loop top -> first chunk computed", nx[105] - nx[0])):
                stages.setdefault(name, []).append(v)
    # the next tile's dequantisation relative to this tile's PV start (P seen, event 14)
    for c in range(ev.shape[0]):
        n = int((ev[c, 12] > 0).sum())
        for it in range(2, n - 1):
            g, nx = ev[c, :, it], ev[c, :, it + 1]
            t0 = g[14]
            rel = {"issuer %d PV block committed" % j: g[24 + j] - t0 for j in range(4)}
            for w in range(8):
                rel["warp %d previous PV seen complete" % w] = nx[88 + w] - t0
            for w in (0, 4):
                for kc in range(5):
                    rel["warp %d chunk step %d arrived" % (w, kc)] = nx[48 + 5 * w + kc] - t0
            rel["slowest warp: tile dequantised, next rows fetched"] = max(nx[32 + w] for w in range(8)) - t0
            for k in range(9):
                rel["issuer 0: next QK chunk %d issued" % k] = nx[112 + k] - t0
            rel["issuer 0: next QK committed"] = nx[12] - t0
            for name, v in rel.items():
                stages.setdefault("t(PV start) + " + name, []).append(v)
    if not period:
        print("no steady tiles traced")
        return
    print(f"decode_main tile period (cycles, median over {len(period)} tiles): {np.median(period):.0f}")
    for k, v in stages.items():
        print(f"  {k:60s} {np.median(v):7.0f}")


def run_trace(args):
    """Per-tile event timeline of the main decode kernel from the trace build
    (-DQMLA_TRACE_BUILD: clock64 stamps at pipeline events of the first eight
    CTAs, written through the buffer given to qmla_trace_set). Stamps are per-SM
    clocks: only differences within one CTA mean anything (event numbers in
    main_trace_summary)."""
    import ctypes

    import numpy as np

    from paper_2609_36760_gb300 import build as B
    lib_path = os.path.join(B.LIBDIR, "libqmla_trace.so")
    srcs = [os.path.join(B.CSRC, f) for f in os.listdir(B.CSRC)] + [os.path.join(B.INCLUDE, "qmla.h")]
    if not os.path.exists(lib_path) or max(map(os.path.getmtime, srcs)) > os.path.getmtime(lib_path):
        lib_path = B.build(trace=True)
    import paper_2609_36760_gb300 as Q
    Q._LIB_PATH = lib_path  # the traced library, loaded before any other call
    L = Q.lib()
    L.qmla_trace_set.argtypes, L.qmla_trace_set.restype = [ctypes.c_void_p], ctypes.c_int
    dev = torch.device("cuda", 0)
    st = Workspace(W.WORKLOADS[args.workload], args.bf16_cache, dev, 4, protect=args.protect, c4r4=args.c4r4,
                   q_tokens=args.q_tokens)
    buf = torch.zeros(TRACE_CTAS * TRACE_EVENTS * TRACE_TILES + 4 * 1024, dtype=torch.int64, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for i in range(3):
        flush.zero_()
        st.step(i)
    L.qmla_trace_set(ctypes.c_void_p(buf.data_ptr()))
    flush.zero_()
    st.step(3)
    torch.cuda.synchronize()
    L.qmla_trace_set(None)
    if Q.read_dev_err(st.err) != 0:
        raise SystemExit(f"device error word {Q.read_dev_err(st.err):#x}")
    t = buf.cpu().numpy()
    np.savez(args.trace, t=t)
    ev = t[:TRACE_CTAS * TRACE_EVENTS * TRACE_TILES].reshape(TRACE_CTAS, TRACE_EVENTS, TRACE_TILES)
    cta = t[TRACE_CTAS * TRACE_EVENTS * TRACE_TILES:].reshape(-1, 4)
    live = cta[cta[:, 0] > 0]
    print(f"CTAs {len(live)}, wall us {(live[:, 1] - live[:, 0]).min() / 1e3:.1f} .. "
          f"{(live[:, 1] - live[:, 0]).max() / 1e3:.1f}, tiles per CTA {live[:, 3].min()} .. {live[:, 3].max()}")
    print(f"raw stamps saved to {args.trace}")
    main_trace_summary(ev)


def main():
    args = parse()
    if args.trace:
        run_trace(args)
        return
    ws_world, rank, local = dist_env()
    if args.impl == "reference":
        run_reference(args, ws_world, rank)
        return
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (the native path has no CPU fallback)")
    run_native(args, ws_world, rank, local)


if __name__ == "__main__":
    main()
