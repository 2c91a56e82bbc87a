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

from eqb_workloads import SHAPES, even_offsets, make_bias, make_grad, make_logits  # noqa: E402

METRIC = "EQB+LEI routing-balance tokens/s per MoE layer; achieved HBM GB/s vs GB300 peak"
ETA, C_NORM = 2e-5, 1.0  # the paper's chosen LEI gain (App. E.3 sweep) and a unit bound


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


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
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


class Step:
    """Device buffers and the launch sequence of one routing-balance step."""

    def __init__(self, T, E, K, M, dev, seed_shift=0):
        import paper_2609_28053_gb300 as eqb
        self.eqb = eqb
        self.T, self.E, self.K, self.M = T, E, K, M
        self.z = make_logits("global", T=T, seed=SHAPES["global"].seed + seed_shift, device=str(dev))
        self.b = make_bias("global", device=str(dev))
        self.g = make_grad("global", T=T, device=str(dev))
        self.off = torch.from_numpy(even_offsets(T, M)).to(dev)
        self.ws = eqb.EqbWorkspace(E, device=dev)
        self.idx = torch.empty((T, K), dtype=torch.int32, device=dev)
        self.tau = torch.empty(T, dtype=torch.float32, device=dev)
        self.loads = torch.zeros((M, E), dtype=torch.int32, device=dev)
        self.b_next = torch.empty(E, dtype=torch.float32, device=dev)
        self.r_global = None
        self.names = ["route_topk", "margin_hist_pass1", "select_pass1", "margin_hist_pass2",
                      "select_pass2", "bias_update", "lei_inject_grad"]

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
        rec(0, lambda: eqb.eqb_route_topk(z, self.b, self.K, self.off, self.idx, self.tau, self.loads,
                                          None, ws.err, stream))
        rec(1, lambda: eqb.eqb_margin_hist_pass1(z, self.tau, ws.hist_hi, ws.err, stream))
        if world > 1:
            torch.distributed.all_reduce(ws.hist_hi)
        rec(2, lambda: eqb.eqb_select_quantile(ws.hist_hi, 1, r, ws.u, ws.rho, None, ws.err, stream))
        rec(3, lambda: eqb.eqb_margin_hist_pass2(z, self.tau, ws.u, ws.hist_lo, stream))
        if world > 1:
            torch.distributed.all_reduce(ws.hist_lo)
        rec(4, lambda: eqb.eqb_select_quantile(ws.hist_lo, 2, r, ws.u, ws.rho, ws.q_hat, ws.err, stream))
        rec(5, lambda: eqb.eqb_bias_update(ws.q_hat, self.b_next, stream))
        rec(6, lambda: eqb.lei_inject_grad(g, self.loads, self.off, self.K, ETA, C_NORM, stream))

    def algorithmic_bytes(self):
        """Bytes the two-pass method must move per step (see the design notes):
        pass 1 reads z (2TE) and writes idx (4TK) and tau (4T); pass 2 reads z
        (2TE) and tau (4T); LEI reads and writes grad (8TE).  Per kernel:"""
        T, E, K = self.T, self.E, self.K
        return {"route_topk": 2 * T * E + 4 * T * K + 4 * T,
                "margin_hist_pass1": 2 * T * E + 4 * T,
                "margin_hist_pass2": 2 * T * E + 4 * T,
                "lei_inject_grad": 8 * T * E,
                "path": 12 * T * E + 8 * T + 4 * T * K}


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


def run_reference(args):
    ws, rank, local = dist_env()
    if rank != 0:
        return
    sh = SHAPES["global"]
    n = args.ref_sample_tokens
    z = make_logits("global", T=n, device="cpu")
    b = make_bias("global", device="cpu")
    g = make_grad("global", T=n, device="cpu")
    for _ in range(args.warmup):
        cpu_oracle_sample(z, b, g, sh.K, n, 32768)
    times = [cpu_oracle_sample(z, b, g, sh.K, n, 32768)[0] for _ in range(args.steps)]
    tot = sum(times)
    value = args.steps * n / tot
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": f"global: T={sh.T} E={sh.E} K={sh.K} M={sh.M}, oracle on a "
                                   f"{n}-token sample per step", "T": sh.T, "E": sh.E, "K": sh.K},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                             "sample": f"first {n} tokens of the workload per step",
                             "host_cores_available": len(os.sched_getaffinity(0))},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--tokens", type=int, default=SHAPES["global"].T)
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--cpu-sample-tokens", type=int, default=131072)
    ap.add_argument("--ref-sample-tokens", type=int, default=32768)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--traffic-json", default=os.path.join(ROOT, "profiles", "traffic.json"))
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)

    world, rank, local = dist_env()
    if world > 1:
        torch.distributed.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    sh = SHAPES["global"]
    T, E, K, M = args.tokens, sh.E, sh.K, max(1, args.tokens // 32768)
    step = Step(T, E, K, M, dev, seed_shift=rank)
    step.r_global = step.eqb.eqb_target_rank(T * world, E, K)
    stream = torch.cuda.current_stream()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        step.run(stream, world)
    barrier()
    err = step.ws.err.item()
    if err:
        raise RuntimeError(f"device flagged {step.eqb.STATUS.get(err, err)}")

    nk = len(step.names)
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(nk)] for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    barrier()
    clocks.start()
    t_start.record(stream)
    for s in range(args.steps):
        step.run(stream, world, events=evs[s])
    t_end.record(stream)
    barrier()
    clk = clocks.stop()
    ms = t_start.elapsed_time(t_end)
    if world > 1:
        tt = torch.tensor([ms], device=dev)
        torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
        ms = tt.item()
    ms_per_step = ms / args.steps
    value = world * T / (ms_per_step / 1e3)

    per_kernel = {}
    for i, name in enumerate(step.names):
        per_kernel[name] = statistics.mean(evs[s][i][0].elapsed_time(evs[s][i][1]) for s in range(args.steps))
    alg = step.algorithmic_bytes()
    peak, peak_kind = measured_peaks()
    dom = max(per_kernel, key=per_kernel.get)
    dom_bytes = alg.get(dom)
    traffic = None
    if os.path.exists(args.traffic_json):
        with open(args.traffic_json) as f:
            tj = json.load(f)
        ent = tj.get(dom)
        if ent and ent.get("T") == T and ent.get("E") == E:
            traffic = ent.get("bytes_per_launch")
    achieved = dom_bytes / (per_kernel[dom] * 1e-3) / 1e9
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "peak_source": peak_kind, "traffic": traffic,
                "algorithmic_bytes": dom_bytes}
    path_gbs = alg["path"] / (ms_per_step * 1e-3) / 1e9
    kernels = {k: {"ms": round(v, 5), "share": round(v / sum(per_kernel.values()), 4),
                   **({"GB/s": round(alg[k] / (v * 1e-3) / 1e9, 1), "frac": round(alg[k] / (v * 1e-3) / 1e9 / peak, 4)}
                      if k in alg else {})} for k, v in per_kernel.items()}

    # ---- end to end through the public API with pinned host buffers
    e2e = None
    if args.e2e_steps > 0:
        z_h = step.z.cpu().pin_memory()
        g_h = step.g.cpu().pin_memory()
        g_out = torch.empty_like(g_h).pin_memory()
        bn_out = torch.empty(E, dtype=torch.float32).pin_memory()
        ld_out = torch.empty((M, E), dtype=torch.int32).pin_memory()
        z_d = torch.empty_like(step.z)
        g_d = torch.empty_like(step.g)
        h2d = z_h.numel() * 2 + g_h.numel() * 4
        d2h = g_out.numel() * 4 + bn_out.numel() * 4 + ld_out.numel() * 4

        def e2e_step():
            z_d.copy_(z_h, non_blocking=True)
            g_d.copy_(g_h, non_blocking=True)
            step.run(stream, world, z=z_d, g=g_d)
            g_out.copy_(g_d, non_blocking=True)
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
        if world > 1:
            tt = torch.tensor([e_ms], device=dev)
            torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
            e_ms = tt.item()
        e2e = {"value": world * T / (e_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e_ms}

    cpu_base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n = min(args.cpu_sample_tokens, T)
        secs, toks = cpu_oracle_sample(step.z, step.b, step.g, K, n, 32768)
        cpu_base = {"value": toks / secs, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                    "sample": f"first {n} tokens of the workload ({max(1, n // 32768)} microbatches): "
                              f"routing, exact quantile of all {E} experts by full sort, bias update, LEI",
                    "seconds": secs, "host_cores_available": len(os.sched_getaffinity(0))}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                "data": "synthetic",
                "config": {"workload": f"global: T={T} E={E} K={K} M={M} per GPU, bf16 logits",
                           "T": T, "E": E, "K": K, "M": M, "eta": ETA, "c": C_NORM,
                           "l2": "inputs larger than L2 (z 1 GiB, grad 2 GiB); no flush",
                           "parallelism": f"dp{world}"},
                "gpu_launches": nk * args.steps,
                "roofline": roofline,
                "path": {"algorithmic_bytes": alg["path"], "GB/s": path_gbs, "frac": path_gbs / peak},
                "kernels": kernels,
                "clocks": clk, "e2e": e2e, "cpu_baseline": cpu_base,
                "elements_per_s": value * E}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
