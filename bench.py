"""Benchmark of the EQB + LEI routing-balance step on GB300.

One step = the whole hot path of one MoE layer on one batch:
  routing (top-K, cutoffs, loads) + coarse margin histogram, pass-1
  selection, fine histogram, pass-2 selection, bias update, and LEI on the
  router-score gradients.  Default workload: T = 2,097,152 tokens, E = 256,
  K = 8, 64 microbatches of 32,768 (synthetic; see eqb_workloads.py).

Prints one JSON line (rank 0).  `value` is tokens/s over all ranks with the
inputs resident in HBM; `e2e` is the same metric through the public API with
pinned host inputs copied in and the result copied out inside the timed
region.  Inputs (z 1 GiB, grad 2 GiB) are larger than the 129 MB L2, so no
flush is needed between timed steps.

Multi-GPU (torchrun): every rank processes its own T-token shard (weak
scaling); the two [E,256] int32 histograms are sum-all-reduced between the
passes, which is Algorithm 1's exchange step.

--impl reference times the CPU oracle (the only reference there is: the
paper publishes no implementation) on a bounded sample per step.
"""
from __future__ import annotations

import argparse
import json
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

from eqb_workloads import (SHAPES, even_offsets, make_bias, make_grad, make_logits,  # noqa: E402
                           prior_batch_logits)

METRIC = "EQB+LEI routing-balance tokens/s per MoE layer; achieved HBM GB/s vs GB300 peak"
ETA, C_NORM = 2e-5, 1.0  # the paper's chosen LEI gain (App. E.3 sweep) and a unit bound


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def allreduce_(t, op=None):
    """t summed (or reduced by op) over the ranks, in place.  NCCL reduces
    device tensors; another backend (gloo) goes through host memory."""
    import torch.distributed as dist
    op = dist.ReduceOp.SUM if op is None else op
    if dist.get_backend() == "nccl":
        dist.all_reduce(t, op=op)
    else:
        h = t.cpu()
        dist.all_reduce(h, op=op)
        t.copy_(h)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.dev), "-lms", "20"], stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return summarize_clock_lines(lines)


def summarize_clock_lines(lines):
    """Median SM clock, maximum SM clock and the throttle reasons seen in
    nvidia-smi rows of ClockSampler.FIELDS (csv, no header, no units)."""
    rows = []
    for line in lines:
        parts = [p.strip() for p in line.split(",")]
        if len(parts) >= 9:
            rows.append(parts)
    if not rows:
        return None
    sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
    mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
    return {"sm_mhz": statistics.median(sm) if sm else None,
            "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


def time_steps(stream, steps, fn, flush=None, sync=torch.cuda.synchronize):
    """Milliseconds of `steps` calls of fn, by CUDA events on `stream`: one
    event pair around the loop, or, with `flush` (a buffer larger than L2),
    one pair around each step, the buffer rewritten before each outside the
    timed region."""
    if flush is None:
        a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_.record(stream)
        for _ in range(steps):
            fn()
        b_.record(stream)
        sync()
        return a_.elapsed_time(b_)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for s_ in range(steps):
        flush.fill_(s_ & 0xff)
        evs[s_][0].record(stream)
        fn()
        evs[s_][1].record(stream)
    sync()
    return sum(a_.elapsed_time(b_) for a_, b_ in evs)


# Workloads whose inputs fit in L2 (129 MB): each step is timed on its own
# after a write of a buffer larger than L2.
SMALL_WORKLOADS = ("tiny", "tie", "mid")


class Step:
    """Device buffers and the launch sequence of one routing-balance step.

    workload 'global': logits resident in HBM (T=2,097,152, E=256, K=8).
    workload 'router': the router projection on the tensor cores first
    (x [T,4096] bf16, W_r [128,4096]), each token routed from the
    projection's accumulators in the same kernel, then the same path on its
    logits; the bias produced by a step is the next step's bias (Eq. 2).
    workloads 'tiny', 'tie', 'mid': the three smaller configurations; the
    'mid' bias is the library's own QB update (eqb_layer_step with b = 0)
    on an independent prior batch of the same distribution."""

    def __init__(self, workload, T, dev, seed_shift=0):
        import paper_2609_28053_gb300 as eqb
        from eqb_workloads import make_router_inputs
        self.eqb = eqb
        self.workload = workload
        sh = SHAPES[workload]
        self.T, self.E, self.K = T, sh.E, sh.K
        self.M = max(1, T // (sh.T // sh.M))
        E = self.E
        if workload == "router":
            self.x, self.W = make_router_inputs(T=T, step=seed_shift, device=str(dev))
            self.d = self.x.shape[1]
            self.z = torch.empty((T, E), dtype=torch.bfloat16, device=dev)
            self.b = torch.zeros(E, dtype=torch.float32, device=dev)
        else:
            self.z = make_logits(workload, T=T, seed=sh.seed + seed_shift, device=str(dev))
            self.b = make_bias(workload, device=str(dev))
            if workload == "mid":
                # b from a prior-step QB update: one step of the library on
                # an independent batch of the same distribution, from b = 0
                prior = prior_batch_logits(workload, T=T, device=str(dev))
                Mp = max(1, T // (sh.T // sh.M))
                offp = torch.from_numpy(even_offsets(T, Mp)).to(dev)
                wsp = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device=dev)
                ldp = torch.zeros((Mp, E), dtype=torch.int32, device=dev)
                bp = torch.empty(E, dtype=torch.float32, device=dev)
                eqb.eqb_layer_step(prior, self.b, self.K, offp, ldp, bp, wsp, mb_offsets_host=even_offsets(T, Mp))
                self.b = bp.clone()
                del prior, wsp
        self.g = make_grad(workload, T=T, device=str(dev))
        self.off = torch.from_numpy(even_offsets(T, self.M)).to(dev)
        self.ws = eqb.EqbWorkspace(E, device=dev)
        self.idx = torch.empty((T, self.K), dtype=torch.int32, device=dev)
        self.tau = torch.empty(T, dtype=torch.float32, device=dev)
        self.loads = torch.zeros((self.M, E), dtype=torch.int32, device=dev)
        self.b_next = torch.empty(E, dtype=torch.float32, device=dev)
        self.r_global = None
        self.off_h = even_offsets(T, self.M)
        self.workspace = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device=dev)
        # The one-call step streams LEI inside the two histogram passes when
        # the [M,E] coefficient table fits its workspace (M * E <= 65,536),
        # and each pass's last block runs that pass's selection; the
        # per-kernel breakdown issues the same work through the separate
        # entry points (the selections as kernels of their own).
        self.fused = self.M * E <= 65536
        self.coef = torch.empty((self.M, E), dtype=torch.float32, device=dev)
        if workload == "router":
            # projection, routing and the coarse histogram in one kernel; the
            # fine pass carries all of LEI
            self.names = (["router_route", "lei_coefficients", "select_pass1", "margin_hist_lei_pass2",
                           "select_pass2", "bias_update"] if self.fused else
                          ["router_route", "select_pass1", "margin_hist_pass2", "select_pass2", "bias_update",
                           "lei_inject_grad"])
        elif self.fused:
            self.names = ["route_topk", "lei_coefficients", "margin_hist_lei_pass1", "select_pass1",
                          "margin_hist_lei_pass2", "select_pass2", "bias_update"]
        else:
            self.names = ["route_topk", "margin_hist_pass1", "select_pass1", "margin_hist_pass2",
                          "select_pass2", "bias_update", "lei_inject_grad"]

    def run_step(self, stream):
        """One step through the one-call entry point eqb_layer_step: routing,
        both histogram passes, selections, the bias update and LEI."""
        eqb = self.eqb
        if self.workload == "router":
            eqb.eqb_router_layer_step(self.x, self.W, self.b, self.K, self.off, self.loads, self.b_next,
                                      self.workspace, z=self.z, tau=self.tau, topk_idx=self.idx,
                                      grad_s=self.g, eta=ETA, c=C_NORM, mb_offsets_host=self.off_h,
                                      r=self.r_global or 0, err_flag=self.ws.err, stream=stream)
            self.b.copy_(self.b_next)  # b^(q+1) routes step q+1
            return
        eqb.eqb_layer_step(self.z, self.b, self.K, self.off, self.loads, self.b_next, self.workspace,
                           tau=self.tau, topk_idx=self.idx, grad_s=self.g, eta=ETA, c=C_NORM,
                           mb_offsets_host=self.off_h, r=self.r_global or 0, err_flag=self.ws.err,
                           stream=stream)

    def run(self, stream, world=1, events=None, z=None, g=None):
        """Enqueue one step.  `events` (optional) is a list of (start, end)
        CUDA event pairs, one per kernel, recorded around each launch."""
        eqb, ws = self.eqb, self.ws
        z = self.z if z is None else z
        g = self.g if g is None else g
        r = self.r_global or eqb.eqb_target_rank(self.T * world, self.E, self.K)

        def rec(i, fn):
            if events is not None:
                events[i][0].record(stream)
            fn()
            if events is not None:
                events[i][1].record(stream)

        ws.hist_hi.zero_()
        ws.hist_lo.zero_()
        ws.err.zero_()
        self.loads.zero_()
        if self.workload == "router":
            rec(0, lambda: eqb.eqb_router_route(self.x, self.W, self.b, self.K, self.off, z, self.idx,
                                                self.tau, self.loads, ws.err, stream, hist_hi=ws.hist_hi))
            if world > 1:
                allreduce_(ws.hist_hi)
            k = 1
            if self.fused:
                rec(1, lambda: eqb.lei_coefficients(self.loads, self.off, self.K, ETA, C_NORM, self.coef, stream))
                k = 2
            rec(k, lambda: eqb.eqb_select_quantile(ws.hist_hi, 1, r, ws.u, ws.rho, None, ws.err, stream))
            if self.fused:
                rec(k + 1, lambda: eqb.eqb_margin_hist_lei(z, self.tau, 2, ws.hist_lo, g, self.coef, self.off, 0,
                                                           self.T, u=ws.u, stream=stream))
            else:
                rec(k + 1, lambda: eqb.eqb_margin_hist_pass2(z, self.tau, ws.u, ws.hist_lo, stream))
            if world > 1:
                allreduce_(ws.hist_lo)
            rec(k + 2, lambda: eqb.eqb_select_quantile(ws.hist_lo, 2, r, ws.u, ws.rho, ws.q_hat, ws.err, stream))
            rec(k + 3, lambda: eqb.eqb_bias_update(ws.q_hat, self.b_next, stream))
            if not self.fused:
                rec(k + 4, lambda: eqb.lei_inject_grad(g, self.loads, self.off, self.K, ETA, C_NORM, stream))
            self.b.copy_(self.b_next)  # b^(q+1) routes step q+1
            return
        rec(0, lambda: eqb.eqb_route_topk(z, self.b, self.K, self.off, self.idx, self.tau,
                                          self.loads, None, ws.err, stream))
        if self.fused:
            th = self.T // 2
            rec(1, lambda: eqb.lei_coefficients(self.loads, self.off, self.K, ETA, C_NORM, self.coef, stream))
            rec(2, lambda: eqb.eqb_margin_hist_lei(z, self.tau, 1, ws.hist_hi, g, self.coef, self.off, 0, th,
                                                   err_flag=ws.err, stream=stream))
        else:
            rec(1, lambda: eqb.eqb_margin_hist_pass1(z, self.tau, ws.hist_hi, ws.err, stream))
        if world > 1:
            allreduce_(ws.hist_hi)
        k = 3 if self.fused else 2
        rec(k, lambda: eqb.eqb_select_quantile(ws.hist_hi, 1, r, ws.u, ws.rho, None, ws.err, stream))
        if self.fused:
            rec(4, lambda: eqb.eqb_margin_hist_lei(z, self.tau, 2, ws.hist_lo, g, self.coef, self.off, th,
                                                   self.T, u=ws.u, stream=stream))
        else:
            rec(3, lambda: eqb.eqb_margin_hist_pass2(z, self.tau, ws.u, ws.hist_lo, stream))
        if world > 1:
            allreduce_(ws.hist_lo)
        k += 2
        rec(k, lambda: eqb.eqb_select_quantile(ws.hist_lo, 2, r, ws.u, ws.rho, ws.q_hat, ws.err,
                                                    stream))
        rec(k + 1, lambda: eqb.eqb_bias_update(ws.q_hat, self.b_next, stream))
        if not self.fused:
            rec(6, lambda: eqb.lei_inject_grad(g, self.loads, self.off, self.K, ETA, C_NORM, stream))

    def launches_per_step(self):
        """Kernels of this library launched by one timed one-call step
        (memsets and torch copies excluded).  Each histogram pass runs its
        own selection in its last block (the fine pass also the bias update).
        Router workload: the projection with routing and the coarse
        histogram, the LEI coefficient table, the pass-1 selection and the
        fine pass carrying LEI: 4.  Otherwise: routing, the coefficient
        table and the two histogram passes carrying the injection: 4.
        Without the table, LEI in its own launch instead: still 4.  (With
        several ranks the histograms are summed between the passes, so the
        step runs as the separate calls of `names`, one kernel each.)"""
        return 4

    def algorithmic_bytes(self):
        """Bytes the two-pass method must move per step (see the design notes):
        pass 1 reads z (2TE) and writes idx (4TK) and tau (4T); pass 2 reads z
        (2TE) and tau (4T); LEI reads and writes grad (8TE); the router
        projection reads x (2Td) and W_r (2Ed) and writes z (2TE), and with
        routing and the coarse histogram in its epilogue leaves only pass 2
        and LEI to read z.  Per kernel:"""
        T, E, K = self.T, self.E, self.K
        th = T // 2
        d = {"route_topk": 2 * T * E + 4 * T * K + 4 * T,
             "margin_hist_pass1": 2 * T * E + 4 * T,
             "margin_hist_pass2": 2 * T * E + 4 * T,
             "lei_inject_grad": 8 * T * E,
             # the fused passes: the pass's z and tau plus its share of grad
             "margin_hist_lei_pass1": 2 * T * E + 4 * T + 8 * th * E,
             "margin_hist_lei_pass2": (2 * T * E + 4 * T + 8 * T * E if self.workload == "router"
                                       else 2 * T * E + 4 * T + 8 * (T - th) * E),
             "path": 12 * T * E + 8 * T + 4 * T * K}
        if self.workload == "router":
            # the projection reads x and W_r and writes z; routing from its
            # accumulators then adds only idx and tau
            d["router_route"] = 2 * T * self.d + 2 * E * self.d + 2 * T * E + 4 * T * K + 4 * T
            d.pop("route_topk")
            # the coarse histogram is counted from the tile just written, so
            # z is read from memory once more, by the fine pass (which carries
            # LEI when the coefficient table fits)
            d["path"] = d["router_route"] + d["margin_hist_pass2"] + d["lei_inject_grad"]
        return d


def dram_traffic(path, kernel, T, E):
    """DRAM bytes (read + write) of one launch of `kernel` at this T and E, as
    recorded from an ncu capture of the same kernel code (lines of
    `kernel T E bytes`; '#' starts a comment); None when not recorded."""
    if not os.path.exists(path):
        return None
    with open(path) as f:
        for line in f:
            parts = line.split("#", 1)[0].split()
            if len(parts) == 4 and parts[0] == kernel and int(parts[1]) == T and int(parts[2]) == E:
                return int(parts[3])
    return None


def cpu_oracle_sample(z_dev, b_dev, g_dev, K, n_tokens, M_per):
    """The oracle, as it stands, on the first n_tokens of the workload:
    routing, the exact quantile of every expert over the sample, the bias
    update and LEI.  Returns (seconds, tokens)."""
    import oracle
    from eqb_workloads import bits
    zb = bits(z_dev[:n_tokens])
    bh = b_dev.cpu().numpy()
    gh = g_dev[:n_tokens].cpu().numpy()
    off = even_offsets(n_tokens, max(1, n_tokens // M_per))
    oracle.build()
    t0 = time.perf_counter()
    st = oracle.eqb_step(zb, bh, K, off)
    oracle.lei(gh, st["loads"], off, K, ETA, C_NORM)
    return time.perf_counter() - t0, n_tokens


def cpu_oracle_router_sample(x_dev, W_dev, g_dev, K, n_tokens):
    """The oracle on the router workload's first n_tokens: the projection
    z_t = W_r x_t in fp64 rounded to bf16, then the routing-balance step."""
    import oracle
    from eqb_workloads import bits
    xb, Wb = bits(x_dev[:n_tokens]), bits(W_dev)
    gh = g_dev[:n_tokens].cpu().numpy()
    off = even_offsets(n_tokens, 1)
    oracle.build()
    t0 = time.perf_counter()
    z64, _ = oracle.router_logits(xb, Wb, np.arange(n_tokens))
    zb = torch.from_numpy(z64.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    st = oracle.eqb_step(zb, np.zeros(Wb.shape[0], np.float32), K, off)
    oracle.lei(gh, st["loads"], off, K, ETA, C_NORM)
    return time.perf_counter() - t0, n_tokens


def run_reference(args):
    ws, rank, local = dist_env()
    if rank != 0:
        return
    wl = args.workload if args.workload != "router" else "global"
    sh = SHAPES[wl]
    n = args.ref_sample_tokens
    per = sh.T // sh.M
    z = make_logits(wl, T=n, device="cpu")
    b = make_bias(wl, device="cpu")
    g = make_grad(wl, T=n, device="cpu")
    for _ in range(args.warmup):
        cpu_oracle_sample(z, b, g, sh.K, n, per)
    times = [cpu_oracle_sample(z, b, g, sh.K, n, per)[0] for _ in range(args.steps)]
    tot = sum(times)
    value = args.steps * n / tot
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": f"{wl}: T={sh.T} E={sh.E} K={sh.K} M={sh.M}, oracle on a "
                                   f"{n}-token sample per step", "T": sh.T, "E": sh.E, "K": sh.K},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                             "sample": f"first {n} tokens of the workload per step",
                             "host_cores_available": len(os.sched_getaffinity(0))},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def e2e_pipelined(step, stream, steps, workload):
    """End to end through the public API, every step's inputs (logits or
    router activations, and the score gradients) copied in from pinned host
    memory and its results (gradients, next bias, loads) copied back, with
    copies and compute on three streams and two device buffer sets, so step
    i's upload, step i-1's compute and step i-2's download overlap.  The
    bias chain of the router workload stays sequential on the compute
    stream (both sets share b)."""
    import copy
    eqb = step.eqb
    other = copy.copy(step)
    if workload == "router":
        other.x = torch.empty_like(step.x)
        other.z = torch.empty_like(step.z)
    else:
        other.z = torch.empty_like(step.z)
    for name in ("g", "idx", "tau", "loads", "b_next", "workspace"):
        setattr(other, name, torch.empty_like(getattr(step, name)))
    other.ws = eqb.EqbWorkspace(step.E, device=step.z.device)
    sets = [step, other]
    srcs = [s_.x if workload == "router" else s_.z for s_ in sets]
    src_h = srcs[0].cpu().pin_memory()
    g_h = step.g.cpu().pin_memory()
    g_out = [torch.empty_like(g_h).pin_memory() for _ in range(2)]
    bn_out = [torch.empty(step.E, dtype=torch.float32).pin_memory() for _ in range(2)]
    ld_out = [torch.empty(tuple(step.loads.shape), dtype=torch.int32).pin_memory() for _ in range(2)]
    h2d = src_h.numel() * src_h.element_size() + g_h.numel() * 4
    d2h = g_out[0].numel() * 4 + bn_out[0].numel() * 4 + ld_out[0].numel() * 4
    s_up, s_down = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_done = [torch.cuda.Event() for _ in range(2)]
    ev_free = [torch.cuda.Event() for _ in range(2)]
    for k in range(2):
        ev_free[k].record(s_down)

    def issue(i):
        k = i % 2
        S = sets[k]
        s_up.wait_event(ev_free[k])
        with torch.cuda.stream(s_up):
            srcs[k].copy_(src_h, non_blocking=True)
            S.g.copy_(g_h, non_blocking=True)
        ev_in[k].record(s_up)
        stream.wait_event(ev_in[k])
        S.run_step(stream)
        ev_done[k].record(stream)
        s_down.wait_event(ev_done[k])
        with torch.cuda.stream(s_down):
            g_out[k].copy_(S.g, non_blocking=True)
            bn_out[k].copy_(S.b_next, non_blocking=True)
            ld_out[k].copy_(S.loads, non_blocking=True)
        ev_free[k].record(s_down)

    issue(0)
    issue(1)
    torch.cuda.synchronize()
    # The host link's rate drops for tens of milliseconds now and then, so
    # the figure is the median of five windows of `steps` steps each (all
    # five are reported).
    windows = []
    for _ in range(5):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(s_up)
        for i in range(steps):
            issue(i)
        b.record(s_down)
        torch.cuda.synchronize()
        windows.append(a.elapsed_time(b) / steps)
    e_ms = statistics.median(windows)
    del other, sets
    return {"value": step.T / (e_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": e_ms, "windows_ms": [round(w, 3) for w in windows],
            "schedule": "upload, compute and download on three streams, two buffer sets"}


def time_call(fn, stream, reps=10):
    """Mean CUDA-event duration (ms) of fn() on `stream`, after one warm-up."""
    fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        fn()
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def extras(step, stream, peak):
    """The comparison rows, timed beside the step (not part of it): the GShard
    gradient (the injection LEI is compared with), MaxVio, the rank-averaged
    and the fixed-resolution estimates of Sec. 2; and the balance each bias
    gives on a fresh batch of the same distribution (Global and Local MaxVio
    after one update)."""
    eqb = step.eqb
    T, E, K, M = step.T, step.E, step.K, step.M
    z, off, dev = step.z, step.off, step.z.device
    shards = even_offsets(T, M)
    lo, width = -4.0, 1.0 / 32
    out = {}

    def row(name, ms, nbytes):
        gbs = nbytes / (ms * 1e-3) / 1e9
        out[name] = {"ms": round(ms, 5), "algorithmic_bytes": nbytes, "GB/s": round(gbs, 1),
                     "frac": round(gbs / peak, 4)}

    g2 = step.g.clone()
    row("gshard_inject_grad", time_call(lambda: eqb.gshard_inject_grad(g2, z, step.loads, off, K, 1e-2, stream),
                                        stream), 10 * T * E)
    del g2
    mv = torch.empty(2, dtype=torch.float64, device=dev)
    out["maxvio"] = {"ms": round(time_call(lambda: eqb.eqb_maxvio(step.loads, off, K, out=mv, stream=stream),
                                           stream), 5)}
    ws_ra = torch.zeros(eqb.eqb_rank_averaged_workspace_bytes(E, M), dtype=torch.uint8, device=dev)
    row("rank_averaged_bias", time_call(lambda: eqb.eqb_rank_averaged_bias(
        z, step.tau, K, shards, ws_ra, stream=stream), stream, reps=3), 2 * (2 * T * E + 4 * T))
    row("fixed_hist_bias", time_call(lambda: eqb.eqb_fixed_hist_bias(
        z, step.tau, K, lo, width, step.workspace, stream=stream), stream), 2 * T * E + 4 * T)

    # Routing with the coarse histogram: the one-read kernel against the two
    # kernels the step uses (routing, then the coarse pass), same outputs.
    if E in (128, 256) and K + 1 <= 16:
        ws = step.ws
        idx2 = torch.empty_like(step.idx)
        tau2 = torch.empty_like(step.tau)
        ld2 = torch.zeros_like(step.loads)

        def two_kernels():
            ws.hist_hi.zero_()
            ld2.zero_()
            eqb.eqb_route_topk(z, step.b, K, off, idx2, tau2, ld2, ws.hist_hi, None, stream)

        def one_kernel():
            ws.hist_hi.zero_()
            ld2.zero_()
            eqb.eqb_route_hist_fused(z, step.b, K, off, idx2, tau2, ld2, ws.hist_hi, None, stream)

        zero_ms = time_call(lambda: (ws.hist_hi.zero_(), ld2.zero_()), stream)
        two = time_call(two_kernels, stream) - zero_ms
        one = time_call(one_kernel, stream) - zero_ms
        out["route_and_coarse_hist"] = {
            "two_kernels_ms": round(two, 5), "one_read_kernel_ms": round(one, 5),
            "two_kernels_bytes": 2 * (2 * T * E) + 4 * T * K + 8 * T,
            "one_read_bytes": 2 * T * E + 4 * T * K + 4 * T}

    # Balance after one update: each bias routes a fresh batch.
    b0 = step.b.clone()
    loads = torch.zeros_like(step.loads)
    tau = torch.empty_like(step.tau)
    eqb.eqb_layer_step(z, b0, K, off, loads, step.b_next, step.workspace, tau=tau, mb_offsets_host=step.off_h,
                       stream=stream)
    biases = {"before": b0, "eqb": step.b_next.clone(),
              "rank_averaged": eqb.eqb_rank_averaged_bias(z, tau, K, shards, ws_ra, stream=stream)[0].clone(),
              "fixed_hist": eqb.eqb_fixed_hist_bias(z, tau, K, lo, width, step.workspace, stream=stream)[0].clone()}
    fresh = make_logits(step.workload, T=T, seed=SHAPES[step.workload].seed + 977, device=str(dev))
    bal = {}
    for name, bb in biases.items():
        loads.zero_()
        eqb.eqb_route_topk(fresh, bb, K, off, None, tau, loads, None, None, stream)
        eqb.eqb_maxvio(loads, off, K, out=mv, stream=stream)
        g_, l_ = mv.tolist()
        bal[name] = {"maxvio_global": round(g_, 4), "maxvio_local": round(l_, 4)}
    # The oracle on a bounded sample of the same workload, one host core.
    import oracle
    from eqb_workloads import bits
    n = min(16384, T)
    per = max(1, T // M)
    zb = bits(z[:n])
    b_h = step.b.cpu().numpy()
    off_n = even_offsets(n, max(1, n // per)) if n >= per else np.array([0, n], np.int64)
    _, tau_n, loads_n = oracle.route(zb, b_h, K, off_n)
    g_n = step.g[:n].cpu().numpy()
    shards_n = even_offsets(n, 4)

    def ocpu(name, fn):
        t0 = time.perf_counter()
        fn()
        secs = time.perf_counter() - t0
        out[name]["cpu_oracle"] = {"tokens_per_s": round(n / secs, 1), "sample_tokens": n, "cores": 1,
                                   "seconds": round(secs, 3)}

    ocpu("gshard_inject_grad", lambda: oracle.gshard(g_n, zb, loads_n, off_n, K, 1e-2))
    ocpu("maxvio", lambda: oracle.maxvio(loads_n, off_n, K))
    ocpu("rank_averaged_bias", lambda: oracle.rank_averaged_bias(zb, tau_n, K, shards_n))
    ocpu("fixed_hist_bias", lambda: oracle.fixed_hist_bias(zb, tau_n, K, lo, width))

    out["maxvio_after_one_update"] = {
        "batch": f"fresh {step.workload} batch, seed +977; biases from the timed batch",
        "rank_averaged_shards": M, "fixed_hist_bins": f"256 x {width} from {lo}", **bal}
    del fresh
    return out


# Steps timed for each of the other workloads in the default run.
OTHER_STEPS = {"tiny": 100, "tie": 50, "mid": 20, "router": 10, "paper": 10, "wide": 20}


def other_workloads(dev, stream, peak, local, skip):
    """The other workloads at their full sizes, each timed the way the
    headline is (the one-call step, three warm-up steps, CUDA events; the
    small ones a step at a time after an L2-evicting write), with its own
    clock record, so that one run of the benchmark measures all of them."""
    out = {}
    for w, n in OTHER_STEPS.items():
        if w == skip:
            continue
        sh = SHAPES[w]
        st = Step(w, sh.T, dev)
        st.r_global = st.eqb.eqb_target_rank(sh.T, st.E, st.K)

        def fn():
            st.run_step(stream)

        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev) if w in SMALL_WORKLOADS else None
        clocks = ClockSampler(local)
        clocks.start()
        time.sleep(0.3)
        ms = time_steps(stream, n, fn, flush) / n
        clk = clocks.stop()
        err = st.ws.err.item()
        gbs = st.algorithmic_bytes()["path"] / (ms * 1e-3) / 1e9
        out[w] = {"ms_per_step": ms, "tokens_per_s": sh.T / (ms * 1e-3), "path_GB/s": round(gbs, 1),
                  "path_frac": round(gbs / peak, 4), "steps": n, "warmup": 3,
                  "T": sh.T, "E": st.E, "K": st.K, "M": st.M,
                  "l2": "per-step eviction" if flush is not None else "inputs larger than L2", "clocks": clk,
                  **({"device_error": st.eqb.STATUS.get(err, err)} if err else {})}
        del st, flush
        torch.cuda.empty_cache()
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="global",
                    choices=["global", "router", "paper", "wide", "tiny", "tie", "mid"])
    ap.add_argument("--tokens", type=int, default=None)
    ap.add_argument("--e2e-steps", type=int, default=8)
    # the oracle's CPU baseline sample: about 10 s of one host core
    ap.add_argument("--cpu-sample-tokens", type=int, default=294912)
    ap.add_argument("--ref-sample-tokens", type=int, default=32768)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true")
    ap.add_argument("--traffic-file", default=os.path.join(ROOT, "profiles", "dram_traffic_per_launch.txt"))
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)

    world, rank, local = dist_env()
    # EQB_BENCH_BACKEND and EQB_BENCH_DEVICE run the multi-rank path with
    # another process-group backend or on a chosen device: two ranks on one
    # GPU through gloo exchange their histograms through host memory, which
    # checks that the path runs and agrees across ranks (not a scaling
    # measurement).
    if world > 1:
        torch.distributed.init_process_group(os.environ.get("EQB_BENCH_BACKEND", "nccl"))
    local = int(os.environ.get("EQB_BENCH_DEVICE", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    sh = SHAPES[args.workload]
    T = args.tokens or sh.T
    step = Step(args.workload, T, dev, seed_shift=rank)
    E, K, M = step.E, step.K, step.M
    step.r_global = step.eqb.eqb_target_rank(T * world, E, K)
    stream = torch.cuda.current_stream()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    one_call = world == 1  # the one-call step keeps its histograms local

    def do_step():
        if one_call:
            step.run_step(stream)
        else:
            step.run(stream, world)

    for _ in range(args.warmup):
        do_step()
    barrier()
    err = step.ws.err.item()
    if err:
        raise RuntimeError(f"device flagged {step.eqb.STATUS.get(err, err)}")

    # On one GPU the one-call step is also captured once as a CUDA graph,
    # whose replay is timed by the same loop after the headline (without the
    # host's per-launch overhead; for the steps timed one at a time a graph
    # launch costs more than it saves).  Several GPUs run the per-pass calls
    # with the all-reduces between them.
    cg, graph_err = None, None
    if one_call:
        try:
            cg = torch.cuda.CUDAGraph()
            gs = torch.cuda.Stream()
            gs.wait_stream(stream)
            torch.cuda.synchronize()
            with torch.cuda.graph(cg, stream=gs, capture_error_mode="relaxed"):
                step.run_step(gs)
            torch.cuda.synchronize()
            cg.replay()  # replay() launches on the current stream
            torch.cuda.synchronize()
        except Exception as exc:  # capture not possible: say why, time the stream loop
            cg, graph_err = None, f"{type(exc).__name__}: {exc}"[:200]

    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev) if args.workload in SMALL_WORKLOADS else None
    clocks = ClockSampler(local)
    barrier()
    clocks.start()
    time.sleep(0.3)  # let the sampler start before the timed region
    ms = time_steps(stream, args.steps, do_step, flush, barrier)
    clk = clocks.stop()
    graph_ms = time_steps(stream, args.steps, cg.replay, flush, barrier) / args.steps if cg is not None else None
    del flush
    err = step.ws.err.item()
    if err:
        raise RuntimeError(f"device flagged {step.eqb.STATUS.get(err, err)}")
    if cg is not None:
        del cg
    if world > 1:
        tt = torch.tensor([ms], device=dev)
        allreduce_(tt, torch.distributed.ReduceOp.MAX)
        ms = tt.item()
    ms_per_step = ms / args.steps
    value = world * T / (ms_per_step / 1e3)
    # Every rank forms the next bias from the same summed histograms, so the
    # ranks must agree bit for bit.
    ranks_agree = None
    if world > 1:
        mine = step.b_next.cpu()
        every = [torch.empty_like(mine) for _ in range(world)]
        torch.distributed.all_gather_object(every, mine)
        ranks_agree = all(torch.equal(mine.view(torch.int32), o.view(torch.int32)) for o in every)
    graph = ({"ms_per_step": graph_ms, "steps": args.steps} if graph_ms is not None else
             {"error": graph_err} if graph_err else None)

    # Per-kernel durations: the same work issued kernel by kernel on one
    # stream, each launch bracketed by CUDA events, in its own timed loop.
    nk = len(step.names)
    ksteps = max(3, min(args.steps, 20))
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(nk)] for _ in range(ksteps)]
    for s_ in range(ksteps):
        step.run(stream, world, events=evs[s_])
    barrier()
    per_kernel = {}
    for i, name in enumerate(step.names):
        per_kernel[name] = statistics.mean(evs[s_][i][0].elapsed_time(evs[s_][i][1]) for s_ in range(ksteps))
    seq_ms = sum(per_kernel.values())
    alg = step.algorithmic_bytes()
    peak, peak_kind = measured_peaks()
    # the roofline's kernel: the slowest of those with algorithmic bytes
    dom = max((k for k in per_kernel if k in alg), key=per_kernel.get)
    dom_bytes = alg.get(dom)
    traffic = dram_traffic(args.traffic_file, dom, T, E)
    achieved = dom_bytes / (per_kernel[dom] * 1e-3) / 1e9
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "peak_source": peak_kind, "traffic": traffic,
                "algorithmic_bytes": dom_bytes}
    path_gbs = alg["path"] / (ms_per_step * 1e-3) / 1e9
    kernels = {k: {"ms": round(v, 5), "share": round(v / sum(per_kernel.values()), 4),
                   **({"GB/s": round(alg[k] / (v * 1e-3) / 1e9, 1), "frac": round(alg[k] / (v * 1e-3) / 1e9 / peak, 4)}
                      if k in alg else {})} for k, v in per_kernel.items()}

    # ---- end to end through the public API with pinned host buffers: the
    # step's inputs (logits, or activations for the router workload, and the
    # score gradients) are copied in and its results (gradients, next bias,
    # loads) copied out inside the timed region.
    e2e = None
    if args.e2e_steps > 0 and world == 1:
        e2e = e2e_pipelined(step, stream, args.e2e_steps, args.workload)
    elif args.e2e_steps > 0:
        src = step.x if args.workload == "router" else step.z
        src_h = src.cpu().pin_memory()
        g_h = step.g.cpu().pin_memory()
        g_out = torch.empty_like(g_h).pin_memory()
        bn_out = torch.empty(E, dtype=torch.float32).pin_memory()
        ld_out = torch.empty((M, E), dtype=torch.int32).pin_memory()
        h2d = src_h.numel() * src_h.element_size() + g_h.numel() * 4
        d2h = g_out.numel() * 4 + bn_out.numel() * 4 + ld_out.numel() * 4

        def e2e_step():
            src.copy_(src_h, non_blocking=True)
            step.g.copy_(g_h, non_blocking=True)
            do_step()
            g_out.copy_(step.g, non_blocking=True)
            bn_out.copy_(step.b_next, non_blocking=True)
            ld_out.copy_(step.loads, non_blocking=True)

        e2e_step()
        barrier()
        a, bq = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(args.e2e_steps):
            e2e_step()
        bq.record(stream)
        barrier()
        e_ms = a.elapsed_time(bq) / args.e2e_steps
        tt = torch.tensor([e_ms], device=dev)
        allreduce_(tt, torch.distributed.ReduceOp.MAX)
        e_ms = tt.item()
        e2e = {"value": world * T / (e_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e_ms, "schedule": "serial on one stream"}

    cpu_base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n = min(args.cpu_sample_tokens if args.workload != "router" else 18432, T)
        if args.workload == "router":
            secs, toks = cpu_oracle_router_sample(step.x, step.W, step.g, K, n)
            what = (f"first {n} tokens: router projection in fp64, routing, exact quantile of all "
                    f"{E} experts by full sort, bias update, LEI")
        else:
            per = T // M
            secs, toks = cpu_oracle_sample(step.z, step.b, step.g, K, n, per)
            what = (f"first {n} tokens of the workload ({max(1, n // per)} microbatches): routing, "
                    f"exact quantile of all {E} experts by full sort, bias update, LEI")
        cpu_base = {"value": toks / secs, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                    "sample": what, "seconds": secs,
                    "host_cores_available": len(os.sched_getaffinity(0))}

    ext = None
    if rank == 0 and world == 1 and not args.no_extras and args.workload != "router":
        ext = extras(step, stream, peak)
    others = None
    if rank == 0 and world == 1 and not args.no_extras and args.tokens is None:
        others = other_workloads(dev, stream, peak, local, args.workload)

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                "data": "synthetic",
                "config": {"workload": (f"router: x [{T},{step.d}] bf16, W_r [{E},{step.d}], "
                                        f"E={E} K={K} M={M} per GPU, bias iterated"
                                        if args.workload == "router" else
                                        f"{args.workload}: T={T} E={E} K={K} M={M} per GPU, bf16 logits"),
                           "T": T, "E": E, "K": K, "M": M, "eta": ETA, "c": C_NORM,
                           "l2": ("each step timed alone after a 512 MiB write that evicts L2 (outside the "
                                  "timed region)" if args.workload in SMALL_WORKLOADS else
                                  "inputs larger than L2 (at least 1 GiB each); no flush"),
                           "parallelism": f"dp{world}"},
                "gpu_launches": (step.launches_per_step() if one_call else len(step.names)) * args.steps,
                "schedule": ("one eqb_layer_step call per step" if one_call
                             else "per-pass calls, histograms all-reduced"),
                "roofline": roofline,
                "path": {"algorithmic_bytes": alg["path"], "GB/s": path_gbs, "frac": path_gbs / peak},
                "kernels": kernels,
                "kernels_sequential_ms": seq_ms,
                "clocks": clk, "e2e": e2e, "cpu_baseline": cpu_base,
                "elements_per_s": value * E, "cuda_graph": graph, "extras": ext,
                "other_workloads": others,
                **({"ranks_agree": ranks_agree} if world > 1 else {})}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
