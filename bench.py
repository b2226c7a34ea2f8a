#!/usr/bin/env python3
"""aTTT update-step benchmark: update tokens/sec on GB300.

One step = one aTTT update (Algorithm 1) of the 32B-class workload, the
largest configuration that one GPU holds:
  Eq. 8/9 weights of the 8,192-token update against the n = 4 history
  (262,144 prior tokens at start), Eq. 10 weighted CE forward + backward
  through the frozen 152,064 x 5,120 bf16 LM head, LoRA rank-64 gradients of
  the q, k, v (one shared input) and o projections, the SGD step on every
  adapter, and the history insert of the update.
The whole step runs in libattt's CUDA kernels, called through the C ABI.
The same run adds, under "extra", the paper's two gradient steps per update
on that workload and the 7B-class single update.

Contract: `python bench.py --gpus N --steps K --warmup W` prints one JSON line.
N > 1 runs N independent replicas (one per GPU, no data-path collective;
value is the sum over ranks).  `--impl reference` times the CPU oracle on the
host cores instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import shutil
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2607_03441_gb300 import workloads as wk  # noqa: E402

METRIC = "aTTT update tokens/sec on 1 GB300 and % of roofline (tensor peak / HBM)"
UNIT = "update tokens/s"
WORKLOAD = "32b"


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16": float(p["bf16_tflops"]),
                "bf16_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "src": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "src": "fallback"}


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        if shutil.which("nvidia-smi") is None:
            return
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                      "--format=csv,noheader,nounits", "-lms", "100"],
                                     stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return self.summarize(lines)

    @staticmethod
    def summarize(lines):
        """Median SM clock, max clock and the throttle reasons seen, from
        `nvidia-smi --query-gpu=QUERY --format=csv,noheader,nounits` lines."""
        rows = []
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
        sm = [r[0] for r in rows]
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(r[1] for r in rows),
                "samples": len(rows), "reasons": reasons}


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

class Update:
    """Device-resident state of one aTTT update of a workload and one step of
    it.  Projections that share an input x (q/k/v; gate/up) form one group
    and one attt_lora_grad call."""

    def __init__(self, wl, dev, max_steps, grad_steps=1):
        import torch
        from paper_2607_03441_gb300 import attt
        self.attt = attt
        self.grad_steps = grad_steps
        self.torch = torch
        self.wl = wl
        self.dev = dev
        if wl.hist_len:
            H = wk.history_tokens(wl)
            self.x_host = wk.update_tokens(wl, H)
        else:  # long episode: the last update against the 31 before it
            ups = wk.long_episode_updates(wl)
            H = np.concatenate(ups[:-1])
            self.x_host = ups[-1]
        dense = wk.dense_inputs(wl)
        self.dense = dense

        def bf(a):
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)

        self.H0 = H
        self.hist = attt.attt_history_create(wl.n, len(H) + wl.L * max_steps)
        attt.attt_history_insert(self.hist, torch.from_numpy(H).to(dev))
        self.x = torch.from_numpy(self.x_host).to(dev)
        self.h = bf(dense["h"])
        self.W = bf(dense["W"])
        self.projs = list(wl.projs)
        self.groups = {}
        for i, p in enumerate(self.projs):
            self.groups.setdefault(p.x_group, []).append(i)
        self.xin = {gname: bf(dense[f"x/{self.projs[idx[0]].name}"]) for gname, idx in self.groups.items()}
        self.dy = [bf(dense[f"dy/{p.name}"]) for p in self.projs]
        self.A32 = [torch.from_numpy(wk.bf16_to_f32(dense[f"A/{p.name}"])).to(dev) for p in self.projs]
        self.B32 = [torch.from_numpy(wk.bf16_to_f32(dense[f"B/{p.name}"])).to(dev) for p in self.projs]
        self.A16 = [bf(dense[f"A/{p.name}"]) for p in self.projs]
        self.B16 = [bf(dense[f"B/{p.name}"]) for p in self.projs]
        self.dA = [torch.empty_like(a) for a in self.A32]
        self.dB = [torch.empty_like(b) for b in self.B32]
        L, d, V, r = wl.L, wl.d, wl.V, wl.r
        self.w = torch.empty(L, dtype=torch.float32, device=dev)
        self.loss = torch.empty(1, dtype=torch.float32, device=dev)
        self.dh = torch.empty(L, d, dtype=torch.float32, device=dev)
        self.ws_ce = torch.empty(attt.attt_ce_workspace_bytes(L, d, V), dtype=torch.uint8, device=dev)
        # The groups' gradients are independent (own x, dy, adapters and outputs): the first group runs
        # on the update's stream and every other one on a side stream of its own, each with its own
        # workspace, so one group's ramp and tail overlap another's streaming.
        self.ws_lora = {gname: torch.empty(attt.attt_lora_workspace_bytes(
            L, self.projs[idx[0]].din, [self.projs[i].dout for i in idx], r), dtype=torch.uint8, device=dev)
            for gname, idx in self.groups.items()}
        self.stream = torch.cuda.current_stream()
        self.side = [torch.cuda.Stream(device=dev) for _ in list(self.groups)[1:]]

    ROWS = ("ngram_weights", "weighted_ce_fwd_bwd", "lora_grad", "lora_step", "history_insert")

    def step(self, events=None, part="all"):
        """One update: the weights, `grad_steps` rounds of Eq. 10, the LoRA
        gradients and the SGD step, then the history insert.  `events`
        (optional) maps each row name to a pair of CUDA events recorded around
        that row's calls (the first round's) on the current stream."""
        a = self.attt

        def mark(name, k, g=0):
            if events is not None and g == 0:
                events[name][k].record()

        if part in ("all", "ngram"):
            mark("ngram_weights", 0)
            a.attt_ngram_weights(self.hist, self.x, self.wl.w_min, out=self.w)
            mark("ngram_weights", 1)
        for g in range(self.grad_steps):
            if part in ("all", "ce"):
                mark("weighted_ce_fwd_bwd", 0, g)
                a.attt_weighted_ce_fwd_bwd(self.h, self.W, self.x, self.w, loss=self.loss, dh=self.dh,
                                           workspace=self.ws_ce)
                mark("weighted_ce_fwd_bwd", 1, g)
            if part in ("all", "lora"):
                mark("lora_grad", 0, g)
                names = list(self.groups)
                main = self.torch.cuda.current_stream() if len(names) > 1 else None
                if main is not None:
                    fork = self.torch.cuda.Event()
                    fork.record(main)
                for k, gname in enumerate(names):
                    idx = self.groups[gname]
                    kw = {}
                    if k > 0:  # a side stream of its own, after everything before the fork
                        self.side[k - 1].wait_event(fork)
                        kw["stream"] = self.side[k - 1]
                    a.attt_lora_grad(self.xin[gname], [self.dy[i] for i in idx], [self.A16[i] for i in idx],
                                     [self.B16[i] for i in idx], self.wl.scale, dAs=[self.dA[i] for i in idx],
                                     dBs=[self.dB[i] for i in idx], workspace=self.ws_lora[gname], **kw)
                if main is not None:
                    for st in self.side:
                        join = self.torch.cuda.Event()
                        join.record(st)
                        main.wait_event(join)
                mark("lora_grad", 1, g)
                mark("lora_step", 0, g)
                for i in range(len(self.projs)):
                    a.attt_lora_step(self.A32[i], self.B32[i], self.dA[i], self.dB[i], wk.LORA_LR, self.A16[i],
                                     self.B16[i])
                mark("lora_step", 1, g)
        if part in ("all", "ngram"):
            mark("history_insert", 0)
            a.attt_history_insert(self.hist, self.x)
            mark("history_insert", 1)


def row_work(wl):
    """Algorithmic work of each row of one update: (kind, amount, unit).
    Bytes count each input read once and each output written once; FLOPs
    count the contractions the method defines."""
    L, V, d, n, r = wl.L, wl.V, wl.d, wl.n, wl.r
    groups = {}
    for p in wl.projs:
        groups.setdefault(p.x_group, []).append(p)
    lora_bytes = 0
    for ps in groups.values():
        lora_bytes += 2 * L * ps[0].din + sum(2 * L * p.dout for p in ps)     # each distinct x once, each dy once
        lora_bytes += sum(6 * p.din * r + 6 * r * p.dout for p in ps)         # A, B in (bf16); dA, dB out (fp32)
    step_elems = sum(p.din * r + r * p.dout for p in wl.projs)
    return {
        # Eq. 8/9: tokens in, one 32 B table sector per probe, weights out
        "ngram_weights": ("hbm", 4 * L + 32 * max(L - n + 1, 0) + 4 * L, "B"),
        # Eq. 10: 4 L V d tensor FLOPs (logits once, dh once)
        "weighted_ce_fwd_bwd": ("tensor", 4.0 * L * V * d, "FLOP"),
        "lora_grad": ("hbm", lora_bytes, "B"),
        # fp32 master + grad read, master written, bf16 copy written
        "lora_step": ("hbm", 14 * step_elems, "B"),
        # Algorithm 1 append: token in and one 32 B sector read + written per new n-gram
        "history_insert": ("hbm", 4 * L + 64 * L, "B"),
    }


def peak_kind(region_ms, clk):
    """Which measured bf16 peak a contraction timed in this region is held
    to: the burst figure (cuBLAS timed alone at full clock) when the timed
    region is shorter than a second and its median SM clock stayed within 3%
    of the maximum; the sustained figure (a seconds-long loop at the power
    cap) otherwise.  Without a clock record the region's length decides."""
    short = region_ms < 1000.0
    if clk is None:
        return "burst" if short else "sustained"
    at_max = clk["sm_mhz"] >= 0.97 * clk["sm_max_mhz"]
    return "burst" if (short and at_max) else "sustained"


def _bf16_peak(peaks, kind):
    return peaks["bf16"] if kind == "burst" else peaks["bf16_sustained"]


def row_report(wl, events, peaks, kind="sustained"):
    out = {}
    work = row_work(wl)
    for name, evs in events.items():
        ms = statistics.mean(a.elapsed_time(b) for a, b in evs)
        amount_kind, amount, _ = work[name]
        if amount_kind == "tensor":
            ach = amount / (ms * 1e-3) / 1e12
            out[name] = {"ms": round(ms, 4), "bound": "tensor", "achieved_tflops": round(ach, 1),
                         "frac": round(ach / _bf16_peak(peaks, kind), 4), "peak_kind": kind,
                         "frac_of_burst": round(ach / peaks["bf16"], 4),
                         "frac_of_sustained": round(ach / peaks["bf16_sustained"], 4), "flop": amount}
        else:
            ach = amount / (ms * 1e-3) / 1e9
            out[name] = {"ms": round(ms, 4), "bound": "hbm", "achieved_gbs": round(ach, 1),
                         "frac": round(ach / peaks["hbm_gbs"], 4), "bytes": int(amount)}
    return out


def _tensor_roofline(achieved, peaks, kind, kernel):
    peak = _bf16_peak(peaks, kind)
    return {"bound": "tensor", "achieved": round(achieved, 1), "peak": peak, "unit": "TFLOP/s",
            "frac": round(achieved / peak, 4), "traffic": None, "kernel": kernel,
            "peak_kind": f"bf16 {kind}, {peaks['src']}", "frac_of_burst": round(achieved / peaks["bf16"], 4),
            "frac_of_sustained": round(achieved / peaks["bf16_sustained"], 4)}


def path_work(wl, grad_steps):
    """Algorithmic FLOPs and bytes of one whole update: the weights and the
    insert once, and per gradient step Eq. 10 (4 L V d; W, h, dh once), the
    LoRA gradients (4 L r (din + dout) per projection; each distinct x and
    each dy once, the adapters) and the SGD step."""
    work = row_work(wl)
    L, V, d = wl.L, wl.V, wl.d
    lora_flops = sum(4.0 * L * wl.r * (p.din + p.dout) for p in wl.projs)
    flops = grad_steps * (work["weighted_ce_fwd_bwd"][1] + lora_flops)
    ce_bytes = 2.0 * V * d + 2.0 * L * d + 4.0 * L * d + 8.0 * L
    nbytes = (work["ngram_weights"][1] + work["history_insert"][1]
              + grad_steps * (ce_bytes + work["lora_grad"][1] + work["lora_step"][1]))
    return flops, nbytes


def path_roofline(wl, grad_steps, ms_per_step, peaks, kind):
    """The whole update against the slower of its FLOPs at the bf16 tensor
    peak and its bytes at the HBM bandwidth (the path roofline)."""
    flops, nbytes = path_work(wl, grad_steps)
    t_tensor = flops / (_bf16_peak(peaks, kind) * 1e12)
    t_hbm = nbytes / (peaks["hbm_gbs"] * 1e9)
    t_roof = max(t_tensor, t_hbm)
    t = ms_per_step * 1e-3
    return {"bound": "tensor" if t_tensor >= t_hbm else "hbm", "flop": flops, "bytes": nbytes,
            "roofline_ms": round(t_roof * 1e3, 4), "ms_per_step": round(ms_per_step, 4),
            "frac": round(t_roof / t, 4), "peak_kind": kind,
            "frac_of_burst": round(max(flops / (peaks["bf16"] * 1e12), t_hbm) / t, 4),
            "frac_of_sustained": round(max(flops / (peaks["bf16_sustained"] * 1e12), t_hbm) / t, 4),
            "achieved_tflops": round(flops / t / 1e12, 1)}


# The sources the Eq. 10 call is built from (its kernels, the contraction
# engine they share, the PTX wrappers and the host-side helpers).
CE_SOURCES = ("ce.cu", "tc_gemm.cuh", "gemm_launch.cuh", "attt_common.cuh", "attt_host.h", "api.cu")


def _sources_sha256() -> str:
    """Hash of the sources of the Eq. 10 call, to tell whether a stored ncu
    capture of that call still describes the kernels that run."""
    h = hashlib.sha256()
    files = [os.path.join(ROOT, "paper_2607_03441_gb300", "csrc", f) for f in CE_SOURCES]
    for f in files:
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def _stored_traffic(wl):
    """DRAM bytes per Eq. 10 call from the committed ncu capture, or None when
    there is none for this workload or the kernels changed since."""
    path = os.path.join(ROOT, "profiles", f"ce_{wl.name}_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    if rec.get("csrc_sha256") != _sources_sha256():
        return None
    return rec.get("traffic_bytes_per_call")


def _ce_roofline(wl, t_ce_ms, peaks, traffic, kind):
    flops = 4.0 * wl.L * wl.V * wl.d
    achieved = flops / (t_ce_ms * 1e-3) / 1e12
    peak = _bf16_peak(peaks, kind)
    return {"bound": "tensor", "achieved": round(achieved, 1), "peak": peak, "unit": "TFLOP/s",
            "frac": round(achieved / peak, 4), "traffic": traffic,
            "kernel": "attt_weighted_ce_fwd_bwd (Eq. 10 fwd+bwd; 4*L*V*d algorithmic FLOPs per call)",
            "peak_kind": f"bf16 {kind}, {peaks['src']}",
            "peak_burst": peaks["bf16"], "frac_of_burst": round(achieved / peaks["bf16"], 4),
            "peak_sustained": peaks["bf16_sustained"],
            "frac_of_sustained": round(achieved / peaks["bf16_sustained"], 4)}


class OracleSample:
    """The CPU oracle on a bounded sample of one update (test infrastructure
    reused as the timed CPU baseline; never on the GPU path)."""

    def __init__(self, wl, dense=None, x=None, H=None):
        import oracle
        oracle.build()
        self.oracle = oracle
        self.wl = wl
        self.H = wk.history_tokens(wl) if H is None else H
        self.x = wk.update_tokens(wl, self.H) if x is None else x
        self.dense = wk.dense_inputs(wl) if dense is None else dense

    def run(self, rows: int, grad_steps: int = 1):
        o, wl, dense = self.oracle, self.wl, self.dense
        sel = np.sort(wk.rng_for(wl.seed, "cpu_sample").choice(wl.L, rows, replace=False)).astype(np.int64)
        t0 = time.perf_counter()
        w = o.ngram_weights(self.H, self.x, wl.n, wl.w_min)
        for _ in range(grad_steps):
            o.ce_rows(dense["h"], dense["W"], self.x, w, sel)
            for p in wl.projs:
                dA, dB = o.lora_grad(dense[f"x/{p.name}"][sel], dense[f"dy/{p.name}"][sel], dense[f"A/{p.name}"],
                                     dense[f"B/{p.name}"], wl.scale)
                o.sgd_step(wk.bf16_to_f32(dense[f"A/{p.name}"]), dA.astype(np.float32), wk.LORA_LR)
                o.sgd_step(wk.bf16_to_f32(dense[f"B/{p.name}"]), dB.astype(np.float32), wk.LORA_LR)
        dt = time.perf_counter() - t0
        desc = (f"{rows} of {wl.L} update tokens of the {wl.name} workload per sample: full Eq. 8/9 weights, "
                f"Eq. 10 lse+dh for {rows} rows over all {wl.V} vocab entries, LoRA grads and SGD for those "
                f"rows" + (f", {grad_steps} times" if grad_steps > 1 else "") + "; fp64 C oracle with OpenMP")
        return dt, {"value": round(rows / dt, 3), "unit": UNIT, "cores": o.num_threads(), "kind": "oracle",
                    "sample": desc + f", {dt:.1f} s"}


def max_over_ranks(vals, pg, device):
    """Element-wise max of `vals` over the ranks of process group module `pg`
    (the slowest rank decides each timing)."""
    import torch
    t = torch.tensor([float(v) for v in vals], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return t.tolist()


def replica_throughput(tokens_per_step, steps, world_size, t_ms):
    """Whole-job update tokens/s of `world_size` independent replicas that each
    ran `steps` updates of `tokens_per_step` tokens within t_ms (the max over
    ranks)."""
    return tokens_per_step * steps * world_size / (t_ms * 1e-3)


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _measure_update(wl, dev, steps, warmup, grad_steps, pg, local, e2e=True):
    """Times `steps` updates of workload `wl` (after `warmup` untimed ones) on
    the device, then (if `e2e`) the same number again with every step's inputs
    copied from pinned host memory and the loss read back.  Returns the
    timings and the per-row CUDA-event report inputs."""
    import torch
    from paper_2607_03441_gb300 import attt
    u = Update(wl, dev, 2 * (warmup + steps) + 4, grad_steps)
    torch.cuda.synchronize()
    for _ in range(warmup):
        u.step()
    torch.cuda.synchronize()
    if attt.attt_device_status() != 0 or attt.attt_history_status(u.hist) != 0:
        raise RuntimeError("device status error after warm-up")

    def barrier():
        if pg is not None:
            pg.barrier()

    # ---------------- device-timed region ----------------
    events = {name: [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                     for _ in range(steps)] for name in Update.ROWS}
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    n0 = attt.attt_kernel_launches()
    e0.record()
    for i in range(steps):
        u.step({k: v[i] for k, v in events.items()})
    e1.record()
    torch.cuda.synchronize()
    n1 = attt.attt_kernel_launches()
    barrier()
    clk = clocks.stop()
    t_ms = e0.elapsed_time(e1)
    if attt.attt_device_status() != 0 or attt.attt_history_status(u.hist) != 0:
        raise RuntimeError("device status error in the timed region")
    res = {"u": u, "t_ms": t_ms, "events": events, "clk": clk, "launches": int(n1 - n0)}
    if not e2e:
        return res

    # ---------------- end to end through host buffers ----------------
    # Every step's inputs (tokens, h, each distinct x, each dy) are copied from
    # pinned host memory into one of two device buffer sets on a copy stream,
    # and the loss is read back every step.  Step i computes on set i % 2 while
    # the inputs of step i + 1 are copied into the other set: the copy of step
    # i + 1 waits until step i - 1 (the set's last user) is done, and step i
    # waits until its own inputs have landed.  Every copy is inside the timed
    # region, the first one included.
    names = ["tokens", "h"] + [f"x/{g}" for g in u.groups] + [f"dy/{p.name}" for p in u.projs]
    host_in = {"tokens": torch.from_numpy(u.x_host).pin_memory(),
               "h": torch.from_numpy(u.dense["h"].view(np.int16)).pin_memory()}
    for gname, idx in u.groups.items():
        host_in[f"x/{gname}"] = torch.from_numpy(u.dense[f"x/{u.projs[idx[0]].name}"].view(np.int16)).pin_memory()
    for p in u.projs:
        host_in[f"dy/{p.name}"] = torch.from_numpy(u.dense[f"dy/{p.name}"].view(np.int16)).pin_memory()
    sets = [{k: torch.empty_like(t, device=dev) for k, t in host_in.items()} for _ in range(2)]

    def use_set(bufs):
        u.x = bufs["tokens"]
        u.h = bufs["h"].view(torch.bfloat16)
        for gname in u.groups:
            u.xin[gname] = bufs[f"x/{gname}"].view(torch.bfloat16)
        for i, p in enumerate(u.projs):
            u.dy[i] = bufs[f"dy/{p.name}"].view(torch.bfloat16)

    loss_host = torch.empty(1, dtype=torch.float32).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = loss_host.numel() * loss_host.element_size()
    cs = torch.cuda.Stream(device=dev)
    main = torch.cuda.current_stream()
    ready = [torch.cuda.Event() for _ in range(steps)]
    done = [torch.cuda.Event() for _ in range(steps)]

    def upload(i):
        with torch.cuda.stream(cs):
            if i >= 2:
                cs.wait_event(done[i - 2])
            for k in names:
                sets[i % 2][k].copy_(host_in[k], non_blocking=True)
            ready[i].record(cs)

    barrier()
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record()
    cs.wait_event(f0)
    upload(0)
    for i in range(steps):
        if i + 1 < steps:
            upload(i + 1)
        main.wait_event(ready[i])
        use_set(sets[i % 2])
        u.step()
        done[i].record(main)
        loss_host.copy_(u.loss, non_blocking=True)
    f1.record()
    torch.cuda.synchronize()
    barrier()
    res.update({"t_e2e": f0.elapsed_time(f1), "h2d": h2d, "d2h": d2h})
    return res


def _workload_desc(wl, hist_tokens, grad_steps):
    return (f"{wl.name}: one aTTT update, L={wl.L} tokens, V={wl.V}, d={wl.d}, n={wl.n}, history {hist_tokens} "
            f"tokens at the start (+L per step), LoRA r={wl.r} on " +
            ", ".join(f"{p.name} {p.din}x{p.dout}" for p in wl.projs) +
            (", one SGD step" if grad_steps == 1 else
             f", {grad_steps} SGD steps (weights and insert once; Eq. 10, LoRA grads and SGD per step)") +
            "; every step re-inserts the same update tokens, so from the second step on the Eq. 8/9 weights see a "
            "fully repeated text")


def run_gpu(args):
    import torch
    from paper_2607_03441_gb300 import attt  # noqa: F401  (fails loudly without the CUDA library)
    from paper_2607_03441_gb300 import build
    ws, rank, local = _dist()
    build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    wl = wk.WORKLOADS[args.workload]
    peaks = _peaks()

    if args.part != "all":
        # one stage alone, for profiling: a single timed loop, no e2e, no baseline
        u = Update(wl, dev, 2 * (args.warmup + args.steps) + 4, args.grad_steps)
        u.w.fill_(1.0)
        for _ in range(args.warmup):
            u.step(part=args.part)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.steps):
            u.step(part=args.part)
        e1.record()
        torch.cuda.synchronize()
        status = attt.attt_device_status()
        u.hist.close()
        return {"part": args.part, "workload": wl.name, "steps": args.steps,
                "ms_per_step": round(e0.elapsed_time(e1) / args.steps, 4), "device_status": status}

    m = _measure_update(wl, dev, args.steps, args.warmup, args.grad_steps, pg, local, e2e=True)
    u = m["u"]
    t_ms, t_e2e = m["t_ms"], m["t_e2e"]
    if pg is not None:
        t_ms, t_e2e = max_over_ranks([t_ms, t_e2e], pg, dev)
    kind = peak_kind(t_ms, m["clk"])
    rows = row_report(wl, m["events"], peaks, kind)
    t_ce = rows["weighted_ce_fwd_bwd"]["ms"]
    value = replica_throughput(wl.L, args.steps, ws, t_ms)
    e2e_value = replica_throughput(wl.L, args.steps, ws, t_e2e)
    hist0 = len(u.H0)
    x_host, dense, H0 = u.x_host, u.dense, u.H0
    u.hist.close()
    del u, m["u"]
    torch.cuda.empty_cache()

    # Extra lines of the same run (one GPU only): the paper's two gradient
    # steps per update on this workload, and the 7B-class single update.
    extras = {}
    if ws == 1 and args.extras:
        gs2 = 2 if args.grad_steps == 1 else 1
        steps2 = max(10, args.steps // 5)
        e = _measure_update(wl, dev, steps2, args.warmup, gs2, None, local, e2e=False)
        k2 = peak_kind(e["t_ms"], e["clk"])
        r2 = row_report(wl, e["events"], peaks, k2)
        extras[f"grad_steps_{gs2}"] = {
            "workload": _workload_desc(wl, hist0, gs2), "value": round(replica_throughput(wl.L, steps2, 1, e["t_ms"]), 1),
            "unit": UNIT, "steps": steps2, "ms_per_step": round(e["t_ms"] / steps2, 4),
            "path_roofline": path_roofline(wl, gs2, e["t_ms"] / steps2, peaks, k2),
            "roofline": _ce_roofline(wl, r2["weighted_ce_fwd_bwd"]["ms"], peaks, None, k2),
            "clocks": e["clk"], "gpu_launches": e["launches"]}
        e["u"].hist.close()
        del e
        torch.cuda.empty_cache()
        if wl.name != "7b":
            w7 = wk.WORKLOADS["7b"]
            e = _measure_update(w7, dev, args.steps, args.warmup, 1, None, local, e2e=False)
            k7 = peak_kind(e["t_ms"], e["clk"])
            r7 = row_report(w7, e["events"], peaks, k7)
            extras["7b"] = {
                "workload": _workload_desc(w7, len(e["u"].H0), 1),
                "value": round(replica_throughput(w7.L, args.steps, 1, e["t_ms"]), 1), "unit": UNIT,
                "steps": args.steps, "ms_per_step": round(e["t_ms"] / args.steps, 4),
                "path_roofline": path_roofline(w7, 1, e["t_ms"] / args.steps, peaks, k7),
                "roofline": _ce_roofline(w7, r7["weighted_ce_fwd_bwd"]["ms"], peaks, _stored_traffic(w7), k7),
                "rows": r7, "clocks": e["clk"], "gpu_launches": e["launches"]}
            e["u"].hist.close()
            del e
            torch.cuda.empty_cache()

    out = None
    if rank == 0:
        cpu = None
        if ws == 1 and args.cpu_rows > 0:
            _, cpu = OracleSample(wl, dense=dense, x=x_host, H=H0).run(args.cpu_rows, args.grad_steps)
        out = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(t_ms / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": _workload_desc(wl, hist0, args.grad_steps),
                       "grad_steps": args.grad_steps,
                       "global_batch": wl.L * ws, "seq_len": wl.L, "parallelism": f"replicas{ws}",
                       "l2": f"inputs larger than L2 (LM head {2 * wl.V * wl.d / 1e9:.2f} GB streamed every step)"},
            "e2e": {"value": round(e2e_value, 1), "unit": UNIT, "h2d_bytes_per_step": m["h2d"],
                    "d2h_bytes_per_step": m["d2h"]},
            "gpu_launches": m["launches"],
            "roofline": _ce_roofline(wl, t_ce, peaks, _stored_traffic(wl), kind),
            "path_roofline": path_roofline(wl, args.grad_steps, t_ms / args.steps, peaks, kind),
            "ce_ms_per_call": round(t_ce, 4),
            "rows": rows,
            "clocks": m["clk"],
            "cpu_baseline": cpu,
            "extra": extras,
        }
    if pg is not None:
        pg.barrier()
        pg.destroy_process_group()
    return out


# ---------------------------------------------------------------------------
# the n-gram stress workload: 8,192 update tokens against a 1,048,576-token
# history, n in {3, 4, 5}, repeated-span fraction in {0, 30, 60, 90}%
# ---------------------------------------------------------------------------

def run_stress(args):
    import torch
    from paper_2607_03441_gb300 import attt
    from paper_2607_03441_gb300 import build
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks = _peaks()
    reps = max(3, args.steps)
    out = {"metric": "n-gram history insert and Eq. 8/9 weights, GB/s of algorithmic bytes vs HBM",
           "workload": "stress: 8,192 update tokens vs a 1,048,576-token history, Zipf(1.1) over 128,256",
           "hbm_peak_gbs": peaks["hbm_gbs"], "reps": reps, "cases": []}
    for n in (3, 4, 5):
        H, _ = wk.stress_case(n, 0.0)
        Hd = torch.from_numpy(H).to(dev)
        h = attt.attt_history_create(n, len(H))
        ins_ms = []
        for _ in range(args.warmup + reps):
            attt.attt_history_reset(h)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            attt.attt_history_insert(h, Hd)
            e1.record()
            torch.cuda.synchronize()
            ins_ms.append(e0.elapsed_time(e1))
        if attt.attt_history_status(h) != 0:
            raise RuntimeError("history status error")
        ins_ms = statistics.median(ins_ms[args.warmup:])
        ins_bytes = 4 * len(H) + 64 * (len(H) - n + 1)
        case = {"n": n, "insert": {"tokens": len(H), "ms": round(ins_ms, 4), "bytes": ins_bytes,
                                   "achieved_gbs": round(ins_bytes / ins_ms / 1e6, 1),
                                   "frac": round(ins_bytes / ins_ms / 1e6 / peaks["hbm_gbs"], 4)},
                "weights": []}
        for frac in (0.0, 0.3, 0.6, 0.9):
            _, x = wk.stress_case(n, frac)
            xd = torch.from_numpy(x).to(dev)
            w = torch.empty(len(x), dtype=torch.float32, device=dev)
            for _ in range(args.warmup):
                attt.attt_ngram_weights(h, xd, 0.05, out=w)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                attt.attt_ngram_weights(h, xd, 0.05, out=w)
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / reps
            wb = 4 * len(x) + 32 * (len(x) - n + 1) + 4 * len(x)
            case["weights"].append({"frac": frac, "tokens": len(x), "ms": round(ms, 5), "bytes": wb,
                                    "achieved_gbs": round(wb / ms / 1e6, 1),
                                    "frac_of_hbm": round(wb / ms / 1e6 / peaks["hbm_gbs"], 4),
                                    "tokens_per_s": round(len(x) / (ms * 1e-3), 1)})
        h.close()
        out["cases"].append(case)
    return out


# ---------------------------------------------------------------------------
# chained episodes: Algorithm 1 with the Sec. 4 / Appendix C schedule, the
# adapted projection feeding the LM head (attt_episode_*)
# ---------------------------------------------------------------------------

def _agent_cuts(L, K):
    """Split an update text of L tokens into the texts of K agent steps."""
    return [round(i * L / K) for i in range(K + 1)]


def episode_flops(ew):
    """Tensor FLOPs of one update: per gradient step the Eq. 10 pair (4 L V d),
    the projection forward and input gradient (2 L din d each, plus the
    rank-r terms) and the adapter gradients (4 L r (din + d))."""
    L, V, din, d, r = ew.L, ew.V, ew.din, ew.d, ew.r
    per_step = 4.0 * L * V * d + 2 * (2.0 * L * din * d + 2.0 * L * r * (din + d)) + 4.0 * L * r * (din + d)
    return ew.grad_steps * per_step


def run_episode(args):
    import torch
    from paper_2607_03441_gb300 import attt
    from paper_2607_03441_gb300 import build
    ws, rank, local = _dist()
    build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    ew = wk.EPISODES[args.workload]
    peaks = _peaks()
    texts = wk.episode_texts(ew)
    dense = wk.episode_dense(ew)
    xs_host = [wk.episode_x(ew, k) for k in range(1, ew.updates + 1)]

    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)

    W0, Wlm = bf(dense["W0"]), bf(dense["W"])
    ep = attt.Episode(W0, Wlm, torch.from_numpy(dense["A0"]).to(dev), torch.from_numpy(dense["B0"]).to(dev),
                      n=ew.n, max_history=ew.hist_len + ew.L * ew.updates, max_update=ew.L, scale=ew.scale,
                      lr=ew.lr, w_min=ew.w_min, grad_steps=ew.grad_steps, cadence=ew.cadence)
    H0 = torch.from_numpy(wk.episode_history(ew)).to(dev)
    tok = [torch.from_numpy(t).to(dev) for t in texts]
    xs = [bf(x) for x in xs_host]
    cuts = _agent_cuts(ew.L, ew.cadence)
    losses = torch.empty(ew.grad_steps, dtype=torch.float32, device=dev)
    dx = torch.empty(ew.grad_steps, ew.L, ew.din, dtype=torch.float32, device=dev)
    state = {"k": 0}

    def start_episode():
        ep.reset()
        if ew.hist_len:
            attt.attt_history_insert(ep.history(), H0)

    def step(tok_k=None, x_k=None):
        """One update: K agent steps, the last of which trains; a new episode
        (reset + prior history) starts after the last update of one."""
        k = state["k"]
        if k == 0:
            start_episode()
        t, x = (tok[k], xs[k]) if tok_k is None else (tok_k, x_k)
        fired = False
        for i in range(ew.cadence):
            fired = ep.agent_step(t[cuts[i]:cuts[i + 1]], x[cuts[i]:cuts[i + 1]], losses=losses, dx=dx)
        assert fired
        state["k"] = (k + 1) % ew.updates

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if attt.attt_device_status() != 0 or attt.attt_history_status(ep.history()) != 0:
        raise RuntimeError("device status error after warm-up")

    def barrier():
        if pg is not None:
            pg.barrier()

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    n0 = attt.attt_kernel_launches()
    e0.record()
    for _ in range(args.steps):
        step()
    e1.record()
    torch.cuda.synchronize()
    n1 = attt.attt_kernel_launches()
    barrier()
    clk = clocks.stop()
    t_ms = e0.elapsed_time(e1)
    if attt.attt_device_status() != 0 or attt.attt_history_status(ep.history()) != 0:
        raise RuntimeError("device status error in the timed region")

    # end to end: each update's text and projection inputs copied from pinned
    # host memory every step, the losses read back every step.  The copies run
    # on a copy stream into two device buffer sets: step i computes on set
    # i % 2 while the inputs of step i + 1 land in the other (the copy of step
    # i + 1 waits until step i - 1, the set's last user, is done; step i waits
    # for its own copy).  Every copy is inside the timed region.
    tok_h = [torch.from_numpy(t).pin_memory() for t in texts]
    xs_h = [torch.from_numpy(x.view(np.int16)).pin_memory() for x in xs_host]
    tok_d = [torch.empty(ew.L, dtype=torch.int32, device=dev) for _ in range(2)]
    x_d = [torch.empty(ew.L, ew.din, dtype=torch.int16, device=dev) for _ in range(2)]
    loss_host = torch.empty(ew.grad_steps, dtype=torch.float32).pin_memory()
    h2d = tok_d[0].numel() * 4 + x_d[0].numel() * 2
    d2h = loss_host.numel() * 4
    cs = torch.cuda.Stream(device=dev)
    main = torch.cuda.current_stream()
    ready = [torch.cuda.Event() for _ in range(args.steps)]
    done = [torch.cuda.Event() for _ in range(args.steps)]

    def upload(i):
        k = i % ew.updates  # the update step i runs (state["k"] starts at 0)
        with torch.cuda.stream(cs):
            if i >= 2:
                cs.wait_event(done[i - 2])
            tok_d[i % 2].copy_(tok_h[k], non_blocking=True)
            x_d[i % 2].copy_(xs_h[k], non_blocking=True)
            ready[i].record(cs)

    state["k"] = 0
    barrier()
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record()
    cs.wait_event(f0)
    upload(0)
    for i in range(args.steps):
        if i + 1 < args.steps:
            upload(i + 1)
        main.wait_event(ready[i])
        step(tok_d[i % 2], x_d[i % 2].view(torch.bfloat16))
        done[i].record(main)
        loss_host.copy_(losses, non_blocking=True)
    f1.record()
    torch.cuda.synchronize()
    barrier()
    t_e2e = f0.elapsed_time(f1)
    # the adapter-drift diagnostic (Sec. 4, Fig. 6) on the last update's rows:
    # 4 L V d algorithmic FLOPs per call (both logit sets once)
    kl = torch.empty(ew.L, dtype=torch.float32, device=dev)
    kl_mean = torch.empty(1, dtype=torch.float32, device=dev)
    x_last = xs[(state["k"] - 1) % ew.updates]
    for _ in range(3):
        ep.drift(x_last, kl, kl_mean)
    torch.cuda.synchronize()
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0.record()
    for _ in range(args.steps):
        ep.drift(x_last, kl, kl_mean)
    g1.record()
    torch.cuda.synchronize()
    t_kl = g0.elapsed_time(g1) / args.steps
    kl_flops = 4.0 * ew.L * ew.V * ew.d + 2 * 2.0 * ew.L * ew.din * ew.d
    if pg is not None:
        t_ms, t_e2e = max_over_ranks([t_ms, t_e2e], pg, dev)

    value = replica_throughput(ew.L, args.steps, ws, t_ms)
    e2e_value = replica_throughput(ew.L, args.steps, ws, t_e2e)
    out = None
    if rank == 0:
        flops = episode_flops(ew)
        ach = flops / (t_ms / args.steps * 1e-3) / 1e12
        cpu = None
        if ws == 1 and args.cpu_rows > 0:
            cpu = _episode_oracle_sample(ew, texts, dense, xs_host, min(args.cpu_rows, 128))[1]
        out = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(t_ms / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": (f"{ew.name}: chained aTTT updates, L={ew.L} tokens in {ew.cadence} agent steps "
                                    f"per update, {ew.updates} updates per episode (reset between episodes), "
                                    f"V={ew.V}, adapter r={ew.r} on a {ew.din}x{ew.d} projection feeding the LM "
                                    f"head, {ew.grad_steps} SGD steps per update with dx, n={ew.n}"),
                       "global_batch": ew.L * ws, "seq_len": ew.L, "parallelism": f"replicas{ws}",
                       "l2": f"inputs larger than L2 (LM head {2 * ew.V * ew.d / 1e9:.2f} GB streamed twice per step)"},
            "e2e": {"value": round(e2e_value, 1), "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": int(n1 - n0),
            "roofline": _tensor_roofline(ach, peaks, peak_kind(t_ms, clk),
                                         "whole update (two Eq. 10 calls, projection forward and dx, adapter grads)"),
            "clocks": clk,
            "cpu_baseline": cpu,
            "kl_drift": {"ms": round(t_kl, 4), "kl_mean": round(kl_mean.item(), 6),
                         "achieved_tflops": round(kl_flops / (t_kl * 1e-3) / 1e12, 1),
                         "frac": round(kl_flops / (t_kl * 1e-3) / 1e12 / _bf16_peak(peaks, peak_kind(t_kl, clk)), 4),
                         "peak_kind": peak_kind(t_kl, clk),
                         "work": "attt_episode_drift: adapted and base projection forward, then the KL through "
                                 "the LM head (4 L V d + 4 L din d FLOPs)"},
        }
    if pg is not None:
        pg.barrier()
        pg.destroy_process_group()
    ep.close()
    return out


def _episode_oracle_sample(ew, texts, dense, xs_host, rows):
    """The oracle's chained update on the first `rows` tokens of the first
    update (all V vocabulary rows, both gradient steps, dx)."""
    import oracle
    oracle.build()
    H = wk.episode_history(ew)
    t0 = time.perf_counter()
    oracle.episode_update(H, texts[0][:rows], xs_host[0][:rows], dense["W0"], dense["W"], dense["A0"],
                          dense["B0"], n=ew.n, w_min=ew.w_min, scale=ew.scale, lr=ew.lr,
                          grad_steps=ew.grad_steps)
    dt = time.perf_counter() - t0
    return dt, {"value": round(rows / dt, 3), "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                "sample": (f"an update of the first {rows} tokens of the {ew.name} workload's first update: Eq. 8/9 "
                           f"weights, {ew.grad_steps} chained gradient steps over all {ew.V} vocab entries with dx; "
                           f"fp64 C oracle with OpenMP, {dt:.1f} s")}


# ---------------------------------------------------------------------------
# a batch of concurrent episodes updated together (attt_batch_*)
# ---------------------------------------------------------------------------

BATCH_EPISODES = 16  # Sec. 4: 16 episodes run concurrently


def run_batch(args):
    """One step = one batched update of 16 episodes (the 7B-class episode's
    shapes): every episode updates on its own 2,048-token text (episode e takes
    text (k + e) mod 16 of the episode workload at step k), two gradient steps
    with dx, one history per episode; all histories and adapters are reset
    after 16 steps."""
    import torch
    from paper_2607_03441_gb300 import attt
    from paper_2607_03441_gb300 import build
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks = _peaks()
    ew = wk.EPISODES["7b-episode"]
    E = BATCH_EPISODES
    texts = wk.episode_texts(ew)
    dense = wk.episode_dense(ew)
    xs_host = [wk.episode_x(ew, k) for k in range(1, ew.updates + 1)]

    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)

    W0, Wlm = bf(dense["W0"]), bf(dense["W"])
    b = attt.Batch(W0, Wlm, torch.from_numpy(dense["A0"]).to(dev), torch.from_numpy(dense["B0"]).to(dev),
                   episodes=E, n=ew.n, max_history=ew.L * ew.updates, max_update=ew.L, scale=ew.scale, lr=ew.lr,
                   w_min=ew.w_min, grad_steps=ew.grad_steps)
    xs = [bf(x) for x in xs_host]
    toks = [torch.from_numpy(t).to(dev) for t in texts]
    # the stacked inputs of each step index, resident before timing
    stacked = []
    for k in range(ew.updates):
        order = [(k + e) % ew.updates for e in range(E)]
        stacked.append((torch.cat([toks[i] for i in order]), torch.cat([xs[i] for i in order])))
    lens = [ew.L] * E
    R = ew.L * E
    losses = torch.empty(E, ew.grad_steps, dtype=torch.float32, device=dev)
    dx = torch.empty(ew.grad_steps, R, ew.din, dtype=torch.float32, device=dev)
    state = {"k": 0}

    def step():
        k = state["k"]
        if k == 0:
            b.reset(-1)
        t, x = stacked[k]
        b.update(t, x, lens, losses=losses, dx=dx)
        state["k"] = (k + 1) % ew.updates

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if attt.attt_device_status() != 0:
        raise RuntimeError("device status error after warm-up")
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(0)
    clocks.start()
    n0 = attt.attt_kernel_launches()
    e0.record()
    for _ in range(args.steps):
        step()
    e1.record()
    torch.cuda.synchronize()
    n1 = attt.attt_kernel_launches()
    clk = clocks.stop()
    if attt.attt_device_status() != 0:
        raise RuntimeError("device status error in the timed region")
    t_ms = e0.elapsed_time(e1)
    value = R * args.steps / (t_ms * 1e-3)
    flops = E * episode_flops(ew)
    ach = flops / (t_ms / args.steps * 1e-3) / 1e12
    out = {"metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": round(t_ms / args.steps, 4), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
           "config": {"workload": (f"7b-batch: {E} concurrent episodes updated together (attt_batch_update), each "
                                   f"L={ew.L} tokens, V={ew.V}, adapter r={ew.r} on a {ew.din}x{ew.d} projection "
                                   f"feeding the LM head, {ew.grad_steps} SGD steps with dx, n={ew.n}; "
                                   f"reset after {ew.updates} steps"),
                      "global_batch": R, "seq_len": ew.L, "parallelism": "replicas1",
                      "l2": "inputs larger than L2 (LM head streamed by every Eq. 10 chunk)"},
           "gpu_launches": int(n1 - n0),
           "roofline": _tensor_roofline(ach, peaks, peak_kind(t_ms, clk),
                                        "whole batched update (Eq. 10 over all rows twice, projection forward and "
                                        "dx, adapter grads)"),
           "clocks": clk}
    b.close()
    return out


# ---------------------------------------------------------------------------
# update-text repetition (Eq. 6), novelty (Eq. 7) and the sequence filter
# ---------------------------------------------------------------------------

def run_texts(args):
    """One step = one episode of update texts through attt_repetition (a reset,
    then one call per update), replayed from a CUDA graph.  Algorithmic bytes
    per call: the text once, plus per word occurrence its key probe (8 B) and
    its mask word read and written (16 B)."""
    import torch
    from paper_2607_03441_gb300 import attt
    from paper_2607_03441_gb300 import build
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks = _peaks()
    tw = wk.TEXT_WORKLOADS[args.workload]
    texts = wk.episode_update_texts(tw)
    nbytes = sum(len(t) for t in texts)
    nwords = sum(len(t.split()) for t in texts)
    dtexts = [torch.frombuffer(bytearray(t), dtype=torch.uint8).to(dev) for t in texts]
    ws = attt.WordSets(tw.updates, nbytes)
    out = torch.empty(tw.updates, 2, dtype=torch.float32, device=dev)
    keep = torch.empty(tw.updates, dtype=torch.int32, device=dev)
    outs = [out[k] for k in range(tw.updates)]
    keeps = [keep[k:k + 1] for k in range(tw.updates)]

    def episode():
        attt.attt_wordsets_reset(ws)
        for k, t in enumerate(dtexts):
            attt.attt_repetition(ws, t, tw.tau, out=outs[k], keep=keeps[k])

    def timed(fn):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        for _ in range(args.steps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / args.steps

    for _ in range(args.warmup):
        episode()
    # the host issues a call in a few microseconds, about as long as a call
    # runs on the device: the device time is taken from a CUDA graph of one
    # episode (the reset and every call, replayed as captured), the
    # host-issued time alongside it
    ms_host = timed(episode)
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream(device=dev)
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cap):
        with torch.cuda.graph(graph, stream=cap):
            episode()
    torch.cuda.current_stream().wait_stream(cap)
    for _ in range(args.warmup):
        graph.replay()
    clocks = ClockSampler(0)
    clocks.start()
    ms = timed(graph.replay)
    clk = clocks.stop()
    if attt.attt_wordsets_status(ws) != 0:
        raise RuntimeError("word-set status error")
    alg = nbytes + 24 * nwords
    ach = alg / (ms * 1e-3) / 1e9
    res = {"metric": "Eq. 6/7 update-text repetition and the sequence filter: update texts/s, GB/s of "
                     "algorithmic bytes vs HBM",
           "value": round(tw.updates / (ms * 1e-3), 1), "unit": "update texts/s", "n_gpus": 1, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True, "data": "synthetic",
           "dtype": "u8",
           "config": {"workload": (f"{tw.name}: {tw.updates} update texts of {tw.words} Zipf(1.1) words over a "
                                   f"{tw.vocab}-word vocabulary, spans copied from the previous text at "
                                   f"{tw.frac_first:.0%}->{tw.frac_last:.0%}, tau {tw.tau}; one step = one episode "
                                   f"(reset + {tw.updates} calls), {nbytes} text bytes, {nwords} words")},
           "gpu_launches": tw.updates * args.steps,  # one repetition_kernel per update, replayed
           "host_issued_ms_per_step": round(ms_host, 4),
           "roofline": {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "frac": round(ach / peaks["hbm_gbs"], 4), "traffic": None,
                        "kernel": "attt_repetition (repetition_kernel, one launch per update), per episode"},
           "clocks": clk,
           "kept": int(keep.sum().item())}
    ws.close()
    return res


# ---------------------------------------------------------------------------
# the reference arm: the CPU oracle on the host cores
# ---------------------------------------------------------------------------

def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return None
    wl = wk.WORKLOADS[args.workload if args.workload in wk.WORKLOADS and args.workload != "stress" else WORKLOAD]
    sample = OracleSample(wl)
    for _ in range(args.warmup):
        sample.run(1)
    t = 0.0
    last = None
    for _ in range(args.steps):
        dt, last = sample.run(args.ref_rows, args.grad_steps)
        t += dt
    value = args.ref_rows * args.steps / t
    return {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * t / args.steps, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{wl.name} (oracle sample of {args.ref_rows} update tokens per step)",
                       "global_batch": wl.L, "seq_len": wl.L, "parallelism": "host cores",
                       "grad_steps": args.grad_steps},
            "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": last["cores"], "kind": "oracle",
                             "sample": last["sample"]},
            "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["attt", "reference"], default="attt")
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=["tiny", "7b", "long", "32b", "stress", "7b-batch"] + sorted(wk.EPISODES)
                    + sorted(wk.TEXT_WORKLOADS),
                    help="'stress' times the n-gram insert and weights on the 1M-token history; "
                         "'*-episode' runs chained updates through attt_episode_*")
    ap.add_argument("--part", default="all", choices=["all", "ce", "lora", "ngram"],
                    help="time one stage alone (profiling aid); 'all' is the benchmark")
    ap.add_argument("--cpu-rows", type=int, default=256, help="rows of the oracle CPU-baseline sample (0: skip)")
    ap.add_argument("--grad-steps", type=int, default=1, choices=range(1, 9), metavar="G",
                    help="gradient steps per update of the single-update workloads (the paper takes 2: "
                         "weights and insert once, Eq. 10, LoRA grads and SGD per step)")
    ap.add_argument("--ref-rows", type=int, default=4, help="rows per step of the reference arm")
    ap.add_argument("--no-extras", dest="extras", action="store_false",
                    help="skip the extra lines (the other gradient-step count and the 7B-class update)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        out = run_reference(args)
    elif args.workload == "stress":
        out = run_stress(args)
    elif args.workload in wk.EPISODES:
        out = run_episode(args)
    elif args.workload in wk.TEXT_WORKLOADS:
        out = run_texts(args)
    elif args.workload == "7b-batch":
        out = run_batch(args)
    else:
        out = run_gpu(args)
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
