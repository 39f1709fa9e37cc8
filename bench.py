"""Benchmark of the fused DBLast draft+verify step on GB300.

One step = one dblast_draft_and_verify call over a batch of N sequences
(prior, codes, vocabulary-head pass with fused softmax statistics, draft
tokens, posterior, target pass, fused verify pass, acceptance and
residual/bonus draws, state update).  Inputs are synthetic and resident in HBM
(W 1.2 GB and target logits 165 MB exceed the 129 MB L2, so no flush is
needed).  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun every rank runs an independent replica on its own GPU (the
sequences are independent units; there is no data-path collective) and rank
0 prints the aggregate.  --impl reference times the fp64 CPU oracle on a
bounded sample (one sequence per step) on the host cores.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "draft+verify blocks/sec and accepted tokens/sec at 1 GB300; % of roofline"
PASS_TIMING_PERIOD = 4
UNIT = "blocks/s"


def job_totals(ms, counts, world, device):
    """Whole-job figures of a replicas run: the slowest rank's time (max over
    ranks) and the counts summed over ranks.  One rank: returned as given."""
    if world <= 1:
        return ms, list(counts)
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    c = torch.tensor([float(x) for x in counts], device=device, dtype=torch.float64)
    dist.all_reduce(c)
    return float(t.item()), [int(x) for x in c.tolist()]


def job_value(units_per_rank, world, steps, ms):
    """The job's throughput: units processed by all ranks over the slowest rank's time."""
    return units_per_rank * world * steps / (ms / 1e3)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"],
                    bf16_sus=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


def work_model(cfg):
    """Algorithmic FLOPs and bytes of one step (low-rank factored head)."""
    V, H, K, r, N, B = (cfg[k] for k in ("V", "H", "K", "r", "N", "B"))
    rr = r + (1 if cfg.get("expander_bias") else 0)
    M = N * B
    el = 2 if cfg["dtype"] == "bf16" else 4
    flop_base = 2.0 * V * H * M
    flop_corr = 2.0 * V * rr * K * M
    flop_codes = 2.0 * M * K * r * H
    byts = (V * H * el + N * (B + 1) * V * el + M * H * el + 2 * K * H * r * el +
            K * H * el + M * (4 * K * 3 + 16))
    return dict(flop=flop_base + flop_corr + flop_codes, flop_draft_pass=flop_base + flop_corr,
                bytes=byts, flop_direct=2.0 * V * H * M * K)


class ClockSampler:
    """nvidia-smi samples during the timed region (median SM clock, reasons)."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for nm, val in zip(names, f[5:9]):
                if val.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "samples": len(sm),
                "reasons": sorted(reasons)}


def cpu_baseline(cfg, head, blk, T, Z_T, budget_s=30.0, mode="soft", top_k=0, top_p=0.0):
    """Time the fp64 oracle, as it stands, on sequences of the workload: with
    the BLAS thread pool as it comes (all host cores), then with one thread."""
    import torch
    from oracle import dblast_oracle as orc
    head_cpu = {k: (None if v is None else v.cpu()) for k, v in head.items()}
    blk_cpu = {"hidden": blk["hidden"].cpu(), "anchor": None, "target": blk["target"].cpu(),
               "has_bonus": blk["has_bonus"]}
    pos = torch.full((cfg["N"],), 37, dtype=torch.int64)
    rnd = torch.zeros(cfg["N"], dtype=torch.int32)

    def run(max_seqs, budget):
        n_done, t0 = 0, time.perf_counter()
        while True:
            orc.draft_and_verify(head_cpu, blk_cpu["hidden"], None, blk_cpu["target"],
                                 blk_cpu["has_bonus"], T, Z_T, 0, pos.numpy(), rnd.numpy(),
                                 seqs=[n_done % cfg["N"]], mode=mode, top_k=top_k, top_p=top_p)
            n_done += 1
            el = time.perf_counter() - t0
            if el > budget or n_done >= max_seqs:
                return n_done, el

    n_done, el = run(4, budget_s / 3)
    single = None
    try:
        from threadpoolctl import threadpool_limits
        with threadpool_limits(limits=1):
            n1, el1 = run(1, budget_s / 3)
        single = {"value": n1 / el1, "unit": UNIT, "threads": 1,
                  "sample": "%d sequence(s), BLAS limited to one thread" % n1}
    except ImportError:
        single = _single_thread_child(cfg, head_cpu, blk_cpu, T, Z_T, mode, top_k, top_p,
                                      budget_s / 3)
    return {"value": n_done / el, "unit": UNIT, "cores": _cpu_threads(),
            "kind": "oracle", "nproc": os.cpu_count(), "cpu_model": _cpu_model(),
            "single_thread": single,
            "sample": "%d sequence(s) of the %s workload (one block each, %s mode), fp64 "
                      "direct form" % (n_done, cfg["name"], mode)}


def _single_thread_child(cfg, head_cpu, blk_cpu, T, Z_T, mode, top_k, top_p, budget):
    """The oracle on one sequence of the same inputs in a child process whose
    BLAS and OpenMP pools are limited to one thread from the start (for hosts
    without threadpoolctl)."""
    import tempfile
    import torch
    with tempfile.TemporaryDirectory() as td:
        path = os.path.join(td, "seq0.pt")
        torch.save({"head": head_cpu, "hidden": blk_cpu["hidden"][:1].clone(),
                    "target": blk_cpu["target"][:1].clone(), "has_bonus": blk_cpu["has_bonus"],
                    "T": T, "Z_T": Z_T, "mode": mode, "top_k": top_k, "top_p": top_p,
                    "budget": budget}, path)
        env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1",
                   MKL_NUM_THREADS="1")
        try:
            out = subprocess.run([sys.executable, os.path.abspath(__file__),
                                  "--oracle-single-thread", path], env=env, capture_output=True,
                                 text=True, timeout=budget * 4 + 120)
            d = json.loads(out.stdout.strip().splitlines()[-1])
        except (OSError, subprocess.SubprocessError, ValueError, IndexError) as e:
            return {"value": None, "why": "single-thread child failed: %s" % type(e).__name__}
    return {"value": d["n"] / d["s"], "unit": UNIT, "threads": 1,
            "sample": "%d sequence(s) in a child process with OPENBLAS/OMP/MKL_NUM_THREADS=1"
                      % d["n"]}


def _oracle_single_thread(path):
    """Child side of _single_thread_child: time the oracle on the saved sequence."""
    import torch
    torch.set_num_threads(1)
    from oracle import dblast_oracle as orc
    d = torch.load(path)
    pos = torch.full((1,), 37, dtype=torch.int64).numpy()
    rnd = torch.zeros(1, dtype=torch.int32).numpy()
    n, t0 = 0, time.perf_counter()
    while True:
        orc.draft_and_verify(d["head"], d["hidden"], None, d["target"], d["has_bonus"], d["T"],
                             d["Z_T"], 0, pos, rnd, seqs=[0], mode=d["mode"], top_k=d["top_k"],
                             top_p=d["top_p"])
        n += 1
        el = time.perf_counter() - t0
        if el > d["budget"] or n >= 1:
            break
    print(json.dumps({"n": n, "s": el}))


def _cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo), or None."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return None


def _cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("num_threads")]
        if n:
            return max(n)
    except Exception:
        pass
    return os.cpu_count()


def run_reference(args, cfg, rank):
    """--impl reference: the oracle on the host cores, one sequence per step."""
    import torch
    import synth
    from oracle import dblast_oracle as orc
    if rank != 0:
        return
    head = synth.make_head(cfg, "cpu")
    blk = synth.make_block(cfg, head, 0, "cpu")
    pos, rnd = synth.initial_state(cfg, "cpu")
    L_total = 0

    def step(i):
        o = orc.draft_and_verify(head, blk["hidden"], None, blk["target"], blk["has_bonus"],
                                 args.T, 1.0, i, pos.numpy(), rnd.numpy(),
                                 seqs=[i % cfg["N"]], mode=args.mode)
        return o[0]["accepted"]

    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        L_total += step(1000 + i)
    el = time.perf_counter() - t0
    v = args.steps / el
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg["name"], "N": cfg["N"], "B": cfg["B"], "K": cfg["K"],
                       "r": cfg["r"], "H": cfg["H"], "V": cfg["V"], "T": args.T,
                       "mode": args.mode, "sample": "one sequence (block) per step"},
            "accepted_tokens_per_s": L_total / el,
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": _cpu_threads(),
                             "kind": "oracle", "nproc": os.cpu_count(),
                             "cpu_model": _cpu_model(),
                             "sample": "one sequence of %s per step" % cfg["name"]},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _timed_steps(step, steps, warmup):
    """CUDA-event time (ms) of `steps` calls of step(k) after `warmup` calls."""
    import torch
    for k in range(warmup):
        step(k)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for k in range(steps):
        step(warmup + k)
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1)


def run_sweep(args):
    """Entropy sweep (K=16, r=32, N=64): per (T, sigma) cell the mean accepted
    length and throughput, next to the K=1 independent-block baseline with the
    same shapes.  One JSON line per cell."""
    import torch
    import synth
    from paper_2608_05448_gb300 import (Head, Workspace, alloc_draft_out, alloc_verify_out,
                                        dblast_draft_and_verify)
    dev = torch.device("cuda", 0)
    for K in (16, 1):
        for sigma in (0.3, 1.0):
            cfg = synth.config("sweep_k16", K=K, sigma=sigma)
            head_t = synth.make_head(cfg, dev)
            blk = synth.make_block(cfg, head_t, 0, dev)
            head = Head.from_dict(head_t)
            ws = Workspace(head, cfg["N"], cfg["B"], True)
            dout = alloc_draft_out(cfg["N"], cfg["B"], K, dev)
            vouts = [alloc_verify_out(cfg["N"], cfg["B"], True, dev)
                     for _ in range(args.warmup + args.steps)]
            for T in (0.7, 1.0, 1.5):
                pos, rnd = synth.initial_state(cfg, dev)

                def step(k):
                    dblast_draft_and_verify(head, ws, blk["hidden"], pos, rnd, T, 1.0, 77 + k,
                                            blk["target"], True, dout=dout, vout=vouts[k])
                ms = _timed_steps(step, args.steps, args.warmup)
                mean_L = float(torch.stack([v["accepted"].float().mean()
                                            for v in vouts[args.warmup:]]).mean())
                # target-block early determinism of the cell, in the bins of App. B
                det = vouts[args.warmup]["determinism"].float().cpu()
                bins = torch.histc(det, bins=5, min=0.0, max=1.0).int().tolist()
                print(json.dumps({"sweep": {"K": K, "r": cfg["r"], "N": cfg["N"], "B": cfg["B"],
                                            "T": T, "sigma": sigma, "mean_accepted_length": mean_L,
                                            "determinism_mean": float(det.mean()),
                                            "determinism_bins_0.2": bins,
                                            "blocks_per_s": cfg["N"] * args.steps / (ms / 1e3),
                                            "accepted_tokens_per_s":
                                                mean_L * cfg["N"] * args.steps / (ms / 1e3),
                                            "ms_per_step": ms / args.steps,
                                            "data": "synthetic"}}), flush=True)
            del head, ws, blk, head_t


def run_determinism(args, cfg):
    """Target-block early determinism (App. B) on the workload's target logits
    [N, B+1, V]: the paper's estimator setting b = 15, M = 20.  One JSON line:
    ms per call (target statistics, 9,600 inverse-CDF draws, reduction) and
    the HBM rate of the one pass over the target."""
    import torch
    import synth
    from paper_2608_05448_gb300 import dblast_target_determinism
    dev = torch.device("cuda", 0)
    head_t = synth.make_head(cfg, dev)
    blk = synth.make_block(cfg, head_t, 0, dev)
    del head_t
    target = blk["target"]
    N, rows, V = target.shape
    b, M = min(15, rows), 20
    from paper_2608_05448_gb300 import lib
    nbytes = lib().dblast_determinism_workspace_bytes(N, rows, b, V, M)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    res = {}

    def step(k):
        res["out"] = dblast_target_determinism(target, b, args.T, M=M, seed=k, ws=ws)
    ms = _timed_steps(step, args.steps, args.warmup) / args.steps
    out = {k: v.cpu() for k, v in res["out"].items()}
    tbytes = target.numel() * target.element_size()
    print(json.dumps({"determinism": {
        "workload": cfg["name"], "N": N, "rows": rows, "V": V, "b": b, "M": M, "T": args.T,
        "ms_per_call": ms, "target_bytes": tbytes,
        "target_pass_gbs": tbytes / (ms * 1e-3) / 1e9,
        "d_exact_mean": float(out["d_exact"].mean()), "d_hat_mean": float(out["d_hat"].mean()),
        "bins_0.2": torch.histc(out["d_exact"], bins=5, min=0.0, max=1.0).int().tolist(),
        "data": "synthetic"}}), flush=True)


def run_al(args, cfg):
    """Training-side objectives, forward only (block NLL and J_AL at tau = 0.1)
    on target blocks of the workload: one JSON line with ms per call and
    blocks/s, with and without the paper's target filter."""
    import numpy as np
    import torch
    import synth
    from paper_2608_05448_gb300 import Head, Workspace, dblast_al_objective
    dev = torch.device("cuda", 0)
    head_t = synth.make_head(cfg, dev)
    blk = synth.make_block(cfg, head_t, 0, dev)
    head = Head.from_dict(head_t)
    N, B = cfg["N"], cfg["B"]
    ws = Workspace(head, N, B, blk["has_bonus"])
    pos, rnd = synth.initial_state(cfg, dev)
    # target blocks: the target's own top tokens, a fixed input of the timed calls
    g = torch.Generator(device=dev).manual_seed(7)
    probs = torch.softmax(blk["target"][:, :B].float() / args.T, dim=-1)
    tokens = torch.multinomial(probs.reshape(-1, probs.shape[-1]), 1, generator=g)
    tokens = tokens.reshape(N, B).int().contiguous()
    del probs
    for top_k, top_p in ((0, 0.0), (20, 0.95)):
        res = {}

        def step(k):
            res["o"] = dblast_al_objective(head, ws, blk["hidden"], pos, rnd, args.T, 1.0, 3,
                                           tokens, blk["target"], blk["has_bonus"], tau=0.1,
                                           top_k=top_k, top_p=top_p)
        ms = _timed_steps(step, args.steps, args.warmup) / args.steps
        o = {k: v.float().cpu() for k, v in res["o"].items()}
        print(json.dumps({"al_objective": {
            "workload": cfg["name"], "N": N, "B": B, "T": args.T, "top_k": top_k,
            "top_p": top_p, "tau": 0.1, "ms_per_call": ms, "blocks_per_s": N / (ms * 1e-3),
            "nll_mean": float(o["nll"].mean()),
            "j_al_mean": float(o["j_al"][torch.isfinite(o["j_al"])].mean()),
            "l_tau_mean": float(o["l_tau"].mean()), "data": "synthetic"}}), flush=True)


def run_serve(args):
    """Serving steps (N=256, B=8 and 32): four rounds with fresh hidden states
    and targets per round and per-sequence state (positions, round counters,
    hence Philox counters) carried on the device.  One JSON line per round."""
    import torch
    import synth
    from paper_2608_05448_gb300 import (Head, Workspace, alloc_draft_out, alloc_verify_out,
                                        dblast_draft_and_verify)
    dev = torch.device("cuda", 0)
    for name in ("serve_b8", "serve_b32"):
        cfg = synth.config(name)
        head_t = synth.make_head(cfg, dev)
        head = Head.from_dict(head_t)
        ws = Workspace(head, cfg["N"], cfg["B"], True)
        dout = alloc_draft_out(cfg["N"], cfg["B"], cfg["K"], dev)
        vout = alloc_verify_out(cfg["N"], cfg["B"], True, dev)
        pos, rnd = synth.initial_state(cfg, dev)
        for rd in range(4):
            blk = synth.make_block(cfg, head_t, rd, dev)
            # the timed call is the round itself; warm-up calls run on copies of the state
            p_w, r_w = pos.clone(), rnd.clone()
            for _ in range(args.warmup):
                dblast_draft_and_verify(head, ws, blk["hidden"], p_w, r_w, 1.0, 1.0, 5,
                                        blk["target"], True, dout=dout, vout=vout)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            dblast_draft_and_verify(head, ws, blk["hidden"], pos, rnd, 1.0, 1.0, 5,
                                    blk["target"], True, dout=dout, vout=vout)
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            L = vout["accepted"].float()
            print(json.dumps({"serve": {"workload": name, "round": rd, "N": cfg["N"],
                                        "B": cfg["B"], "ms": ms,
                                        "blocks_per_s": cfg["N"] / (ms / 1e3),
                                        "mean_accepted_length": float(L.mean()),
                                        "min_accepted": int(L.min()), "max_accepted": int(L.max()),
                                        "emitted_tokens": int(vout["n_emitted"].sum()),
                                        "mean_position": float(pos.double().mean()),
                                        "data": "synthetic"}}), flush=True)
            del blk
        del head, ws, head_t


def main():
    if len(sys.argv) == 3 and sys.argv[1] == "--oracle-single-thread":
        _oracle_single_thread(sys.argv[2])
        return
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="qwen3_8b_b32")
    ap.add_argument("--T", type=float, default=1.0)
    ap.add_argument("--kernels", default="auto", choices=["auto", "simt", "tcgen05"])
    ap.add_argument("--top-k", type=int, default=0,
                    help="target filter: top-k (0 = off; the paper uses 20)")
    ap.add_argument("--top-p", type=float, default=0.0,
                    help="target filter: top-p (0 = off; the paper uses 0.8 / 0.95)")
    ap.add_argument("--mode", default="soft", choices=["soft", "greedy"],
                    help="draft tokens sampled from the z-hat branch (soft) or the "
                         "greedy-branch decoder")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=None)
    ap.add_argument("--sweep", action="store_true",
                    help="entropy-sweep report (K=16 vs K=1 cells), one JSON line per cell")
    ap.add_argument("--determinism", action="store_true",
                    help="target-block early determinism report (b = 15, M = 20), one JSON line")
    ap.add_argument("--al", action="store_true",
                    help="training-side objectives (block NLL, J_AL), forward only, one JSON line "
                         "per filter setting")
    ap.add_argument("--serve", action="store_true",
                    help="serving report (N=256, B=8/32, four rounds), one JSON line per round")
    ap.add_argument("--n-seqs", type=int, default=None,
                    help="override the number of sequences N (smaller cases for profiler captures)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    import synth
    cfg = synth.config(args.config, **({"N": args.n_seqs} if args.n_seqs else {}))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, cfg, rank)
        return
    if args.sweep or args.serve or args.determinism or args.al:
        import torch
        torch.cuda.set_device(0)
        if args.determinism:
            run_determinism(args, cfg)
        if args.al:
            run_al(args, cfg)
        if args.sweep:
            run_sweep(args)
        if args.serve:
            run_serve(args)
        return

    import torch
    import torch.distributed as dist
    torch.cuda.set_device(local)
    if world > 1:
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2608_05448_gb300 import (Head, Workspace, alloc_draft_out, alloc_verify_out,
                                        dblast_draft_and_verify, dblast_stats_get,
                                        dblast_stats_reset)
    peaks = load_peaks()
    dev = torch.device("cuda", local)
    head_t = synth.make_head(cfg, dev)
    blk = synth.make_block(cfg, head_t, 0, dev)
    N, B = cfg["N"], cfg["B"]
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    head = Head.from_dict(head_t)
    torch.cuda.synchronize()
    prep_ms = 1e3 * (time.perf_counter() - t0)
    ws = Workspace(head, N, B, blk["has_bonus"])
    pos, rnd = synth.initial_state(cfg, dev)
    K_steps = args.steps
    dout = alloc_draft_out(N, B, cfg["K"], dev, args.mode)
    vouts = [alloc_verify_out(N, B, blk["has_bonus"], dev) for _ in range(K_steps)]
    seed = 1234 + 7919 * rank

    def step(vout):
        dblast_draft_and_verify(head, ws, blk["hidden"], pos, rnd, args.T, cfg["Z_T"], seed,
                                blk["target"], blk["has_bonus"], impl=args.kernels,
                                dout=dout, vout=vout, mode=args.mode, top_k=args.top_k,
                                top_p=args.top_p)

    for _ in range(args.warmup):
        step(vouts[0])
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    # CUDA events around the passes of every PASS_TIMING_PERIOD-th timed step
    # only: an event between two kernels keeps the later one from starting
    # early, so timing every step would slow the step it measures
    dblast_stats_reset(PASS_TIMING_PERIOD)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record()
    for k in range(K_steps):
        step(vouts[k])
    ev1.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    st = dblast_stats_get()
    accepted = sum(int(v["accepted"].sum()) for v in vouts)
    emitted = sum(int(v["n_emitted"].sum()) for v in vouts)
    # decisions the kernels flagged as within the tie tolerance of their
    # threshold (tie_flags), counted over the timed steps
    flags = torch.stack([v["tie_flags"] for v in vouts]).cpu()
    tie_seqs = int(((flags & 0xFF) != 0).sum())
    near_seqs = int((flags != 0).sum())
    tie_bits = {name: int(((flags & bit) != 0).sum()) for name, bit in
                (("zhat", 1), ("draft", 2), ("accept", 4), ("residual_bonus", 8),
                 ("residual_mass", 16), ("top_p", 32))}

    # the workload's other temperature (the 8B batched workload is quoted at
    # T = 0.6 and 1.0): the same timed loop on the same inputs
    other_T = None
    T2 = 0.6 if (cfg["name"] == "qwen3_8b_b32" and args.T != 0.6) else None
    if T2 is not None:
        pos2, rnd2 = synth.initial_state(cfg, dev)

        def step2(k):
            dblast_draft_and_verify(head, ws, blk["hidden"], pos2, rnd2, T2, cfg["Z_T"], seed,
                                    blk["target"], blk["has_bonus"], impl=args.kernels,
                                    dout=dout, vout=vouts[k % K_steps], mode=args.mode,
                                    top_k=args.top_k, top_p=args.top_p)
        ms2 = _timed_steps(step2, K_steps, args.warmup)
        acc2 = sum(int(v["accepted"].sum()) for v in vouts)
        ms2, (acc2,) = job_totals(ms2, (acc2,), world, dev)
        other_T = {"T": T2, "ms_per_step": ms2 / K_steps,
                   "value": job_value(N, world, K_steps, ms2),
                   "accepted_tokens_per_s": acc2 / (ms2 / 1e3),
                   "mean_accepted_length": acc2 / (N * world * K_steps)}
    ms, (accepted, emitted) = job_totals(ev0.elapsed_time(ev1), (accepted, emitted), world, dev)
    ms_step = ms / K_steps
    value = job_value(N, world, K_steps, ms)

    # end to end through the public API with host buffers (pinned), per step:
    # H2D of hidden + target, the call, D2H of the per-sequence results.  The
    # inputs of step k+1 are copied on a second stream while step k runs
    # (two device buffers); every copy and every call lie between e0 and e1.
    e2e_steps = args.e2e_steps or K_steps
    h_host = blk["hidden"].cpu().pin_memory()
    t_host = blk["target"].cpu().pin_memory()
    # the per-sequence results live in one device buffer (segments 16-byte
    # aligned), so one device-to-host copy reads them back each step
    def seg(n):
        return (n + 3) // 4 * 4
    sizes = [seg(N), seg(N), seg(N * (B + 1)), seg(N)]
    offs = [sum(sizes[:j]) for j in range(4)]
    res_dev = torch.empty(sum(sizes), dtype=torch.int32, device=dev)
    vout_e2e = dict(vouts[0])
    vout_e2e["accepted"] = res_dev[offs[0]:offs[0] + N]
    vout_e2e["n_emitted"] = res_dev[offs[1]:offs[1] + N]
    vout_e2e["emitted"] = res_dev[offs[2]:offs[2] + N * (B + 1)].view(N, B + 1)
    vout_e2e["exp_len"] = res_dev[offs[3]:offs[3] + N].view(torch.float32)
    res_host = torch.empty_like(res_dev, device="cpu").pin_memory()
    h_dev = [torch.empty_like(blk["hidden"]) for _ in range(2)]
    t_dev = [torch.empty_like(blk["target"]) for _ in range(2)]
    h2d = h_host.numel() * h_host.element_size() + t_host.numel() * t_host.element_size()
    d2h = res_host.numel() * res_host.element_size()
    main = torch.cuda.current_stream()
    cstream = torch.cuda.Stream()
    copied = [torch.cuda.Event() for _ in range(2)]
    freed = [torch.cuda.Event() for _ in range(2)]
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(main)

    def copy_in(b, after=None):
        cstream.wait_event(after if after is not None else e0)
        with torch.cuda.stream(cstream):
            h_dev[b].copy_(h_host, non_blocking=True)
            t_dev[b].copy_(t_host, non_blocking=True)
            copied[b].record(cstream)

    copy_in(0)
    for k in range(e2e_steps):
        b = k & 1
        if k + 1 < e2e_steps:
            copy_in(b ^ 1, freed[b ^ 1] if k >= 1 else None)
        main.wait_event(copied[b])
        dblast_draft_and_verify(head, ws, h_dev[b], pos, rnd, args.T, cfg["Z_T"], seed, t_dev[b],
                                blk["has_bonus"], impl=args.kernels, dout=dout, vout=vout_e2e,
                                mode=args.mode, top_k=args.top_k, top_p=args.top_p)
        freed[b].record(main)
        res_host.copy_(res_dev, non_blocking=True)
    e1.record(main)
    torch.cuda.synchronize()
    ems, _ = job_totals(e0.elapsed_time(e1), (), world, dev)
    e2e_value = job_value(N, world, e2e_steps, ems)

    if rank == 0:
        wm = work_model(cfg)
        draft_ms = st["draft_pass_ms"] / max(1, st["timed_draft"])
        verify_ms = st["verify_pass_ms"] / max(1, st["timed_verify"])
        achieved = wm["flop_draft_pass"] / (draft_ms * 1e-3) / 1e12
        t_roof = max(wm["flop"] / (peaks["bf16"] * 1e12), wm["bytes"] / (peaks["hbm"] * 1e9))
        traffic = None
        # DRAM bytes per draft-pass launch from the committed ncu summary, used
        # only while the kernel source is the one that was profiled
        tr_path = os.path.join(ROOT, "profiles", "draft_pass_%s_traffic.json" % cfg["name"])
        if args.mode == "greedy":
            tr_path = os.path.join(ROOT, "profiles", "draft_pass_greedy_%s_traffic.json" % cfg["name"])
        elif args.top_k > 0 or 0.0 < args.top_p < 1.0:
            tr_path = ""  # with a filter the soft pass also reads the target: not captured
        if tr_path and os.path.exists(tr_path) and st["tc_launches"] > 0 and not args.n_seqs:
            d = json.load(open(tr_path))
            src = os.path.join(ROOT, d.get("source", ""))
            if os.path.exists(src):
                hsh = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
                if hsh == d.get("source_sha256_16"):
                    traffic = d.get("bytes_per_launch")
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": K_steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if cfg["dtype"] == "bf16" else "f32", "data": "synthetic",
            "config": {"workload": cfg["name"], "N": N, "B": B, "K": cfg["K"], "r": cfg["r"],
                       "H": cfg["H"], "V": cfg["V"], "T": args.T, "Z_T": cfg["Z_T"],
                       "sigma": cfg["sigma"], "mode": args.mode, "top_k": args.top_k,
                       "top_p": args.top_p,
                       "kernels": "tcgen05" if st["tc_launches"] > 0 else "simt",
                       "parallelism": "replicas" if world > 1 else "single",
                       "l2": "no flush: inputs larger than L2 (W %.2f GB, target %.0f MB)" % (
                           cfg["V"] * cfg["H"] * 2 / 1e9,
                           N * (B + 1) * cfg["V"] * 2 / 1e6)},
            "accepted_tokens_per_s": accepted / (ms / 1e3),
            "emitted_tokens_per_s": emitted / (ms / 1e3),
            "mean_accepted_length": accepted / (N * world * K_steps),
            "roofline_step": {"t_roofline_ms": 1e3 * t_roof, "frac": 1e3 * t_roof / ms_step,
                              "flop": wm["flop"], "bytes": wm["bytes"],
                              "flop_direct_form": wm["flop_direct"],
                              "peak_source": peaks["source"]},
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16"],
                         "unit": "TFLOP/s", "frac": achieved / peaks["bf16"],
                         "traffic": traffic, "kernel": "draft pass",
                         "ms_per_launch": draft_ms, "timed_launches": int(st["timed_draft"]),
                         "timing": "CUDA events on the launching stream around the draft "
                                   "pass of every %dth timed step" % PASS_TIMING_PERIOD},
            "verify_pass_ms": verify_ms,
            "ties": {"sequences_flagged_per_step": tie_seqs / K_steps,
                     "sequences_flagged": tie_seqs, "sequences": N * K_steps,
                     "by_kind": tie_bits,
                     "sequences_near_per_step": near_seqs / K_steps,
                     "what": "sequences whose step took a decision within 1e-6 of its "
                             "threshold by the kernels' arithmetic (tie bits), and within "
                             "1e-6 plus the kernels' precision allowance (near bits), over "
                             "the timed steps"},
            "prep_ms": prep_ms,
            "gpu_launches": int(st["kernel_launches"]),
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                    "overlap": "inputs of step k+1 copied on a second stream during step k"},
            "clocks": clk,
        }
        if other_T is not None:
            other_T["roofline_frac"] = 1e3 * t_roof / other_T["ms_per_step"]
            line["T%.1f" % other_T["T"]] = other_T
        if world == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(cfg, head_t, blk, args.T, cfg["Z_T"],
                                                mode=args.mode, top_k=args.top_k,
                                                top_p=args.top_p)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
