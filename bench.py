"""Benchmark: packed-ensemble training throughput on GB300.

One step = one pass of the whole training path over one batch: gather,
forward through every member, per-member loss, backward, per-member AdamW.
Metric: member-samples/s = (active members) x (batch rows) x steps / time.

  python bench.py [--gpus N --steps K --warmup W --workload medium]
  python bench.py --impl reference ...   # the CPU fp64 oracle on host cores

Under torchrun (N > 1) every rank trains its own full pack (members are
independent; no collective on the data path), so scaling is weak and the
reported value is the sum over ranks of member-samples / max-over-ranks time.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from workloads import SEED_HP, SEED_INIT, WORKLOADS, make_data, sample_emb, sample_hparams  # noqa: E402

METRIC = "member-samples/sec (fwd+bwd+AdamW)"

# DRAM bytes (read + write) per step of the dominant kernels, from ncu captures of
# the current kernels (summaries in profiles/; the wide figure is scaled from its
# first 8 members by GEMM flops).  A workload without a capture reports null.
DRAM_TRAFFIC = {
    ("medium", "k_tc_gemm"): 252.0e6,
    ("medium", "k_adamw"): 607.7e6,
    ("wide", "k_tc_gemm"): 3.589e9,
}
UNIT = "member-samples/s"


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


def muon_lrs(m):
    """Per-member Muon learning rates, LogUniform[1e-3, 1e-1] (seed 101)."""
    rng_m = np.random.default_rng(SEED_HP + 100)
    return np.exp(rng_m.uniform(math.log(1e-3), math.log(1e-1), m)).astype(np.float32)


def in0_of(wl, emb, i):
    """Member i's first-layer input width (d_in d_emb with embeddings)."""
    return wl.d_in * (int(emb["d_emb"][i]) if emb is not None else 1)


def work_per_step(wl, hp, B, emb=None):
    """Algorithmic work of one step, from the shapes (no padding):
    matrix-product flops (forward 2, dgrad 2 except layer 0 -- with
    embeddings layer 0 too, for dE --, wgrad 2 per MAC) and the parameter
    count of the AdamW bytes (read p, g, m, v; write p, m, v fp32 + the bf16
    copy), embeddings included."""
    flops = 0.0
    n_params = 0
    for i, (L, w) in enumerate(zip(hp["depth"], hp["width"])):
        L, w = int(L), int(w)
        in0 = in0_of(wl, emb, i)
        macs_fwd = in0 * w + (L - 1) * w * w
        macs_dgrad = (L - 1) * w * w + (in0 * w if emb is not None else 0)
        flops += 2.0 * B * (2 * macs_fwd + macs_dgrad)
        n_params += in0 * w + w + (L - 1) * (w * w + w) + wl.d_out * w + wl.d_out
        if emb is not None:
            n_params += wl.d_in * (4 * int(emb["d_emb"][i]) - 2)
    return flops, n_params


def max_over_ranks(value, dist, device):
    """The largest of every rank's `value` (the job's timed region ends when
    its slowest rank ends)."""
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, members, batch, steps, ms_total):
    """Whole-job member-samples/s: every rank trains its own pack of
    `members` members on `batch` rows per step (weak scaling)."""
    return world * members * batch * steps / (ms_total / 1000.0)


def workload_desc(wl, B):
    return (f"{wl.name}: {wl.task}, m={wl.m} members, depth U{{{wl.depth[0]}..{wl.depth[1]}}}, width multiples of "
            f"{wl.width[2]} in [{wl.width[0]},{wl.width[1]}], dropout U[{wl.dropout[0]},{wl.dropout[1]}], "
            f"d_in={wl.d_in}, d_out={wl.d_out}, batch={B}, n_train={wl.n_train}")


class ClockSampler:
    """nvidia-smi clock / throttle samples during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu_id}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not getattr(self, "out", ""):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm, smax, reasons = [], [], set()
        names = ["active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                smax.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names[1:], f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def predict_flops(wl, hp, n_rows, emb=None):
    """Matrix-product flops of one forward without dropout of every member
    over n_rows rows (hidden layers and head)."""
    f = 0
    for i, (L, w) in enumerate(zip(hp["depth"], hp["width"])):
        L, w = int(L), int(w)
        f += in0_of(wl, emb, i) * w + (L - 1) * w * w + w * wl.d_out
    return 2.0 * n_rows * f


def time_online_epoch(tp, torch, pack, wl, hp, d, X, y, idx_all, stream, loss, n_epochs=6, steps_between=8,
                      m_ens=32, p_base=16, p_ens=32, score="loss", emb=None):
    """Wall time of the online ensemble's epoch end (Sec. 3.5: predict the
    members on the validation rows, greedy selection over the pool, member
    snapshots, patience bookkeeping) on the workload's full validation set,
    with a few training steps between epoch ends so that states change.  The
    call synchronises, so it is timed on the host around a synchronised
    stream; the prediction share comes from the pack's CUDA-event profile."""
    X_val, y_val = d["X_val"], d["y_val"]
    on = tp.OnlineEnsemble(pack, X_val.shape[0], score, m_ens, p_base, p_ens)
    B = wl.batch
    times, pred_ms = [], []
    s_next = 50_000
    for e in range(n_epochs + 1):
        for k in range(steps_between):
            pack.train_step(X, idx_all[k % idx_all.shape[0]], y, s_next, loss)
            s_next += 1
        torch.cuda.synchronize()
        pack.profile_enable(True)
        pack.profile_read(reset=True)
        t0 = time.perf_counter()
        on.epoch(X_val, y_val)
        dt = (time.perf_counter() - t0) * 1000.0
        prof = pack.profile_read(reset=True)
        pack.profile_enable(False)
        if e > 0:      # the first call warms up
            times.append(dt)
            pred_ms.append(prof["predict"][0] + prof["fwd"][0])
    info = on.info()
    on.close()
    pack.set_active(np.ones(wl.m, dtype=np.uint8))
    ms = float(np.median(times))
    pm = float(np.median(pred_ms))
    n_val = int(X_val.shape[0])
    pool = info["n_pool"]
    sel_bytes = m_ens * pool * n_val * wl.d_out * 4.0
    return {"ms": ms, "predict_ms": pm, "select_and_rest_ms": ms - pm, "n_val": n_val, "m_ens": m_ens, "score": score,
            "pool": pool, "n_best": info["n_best"], "epochs_timed": len(times),
            "predict_tflops": predict_flops(wl, hp, n_val, emb) / (pm / 1e3) / 1e12,
            "select_candidate_bytes": sel_bytes,
            "note": "epoch-end cost once per epoch of %d steps; predictions on the full validation set"
                    % -(-wl.n_train // B)}


def cpu_baseline(wl, hp, data_np, B, budget_s=20.0, stacked=False, emb=None, lr_muon=None):
    """The oracle as it stands, on the host cores, on a bounded sample of the
    same workload: the first k members (independent of the others), timed
    over whole steps until about budget_s seconds of CPU work (stacked: a
    batch per member; emb: the members' periodic embeddings; lr_muon: Muon
    for the hidden weights with these per-member learning rates)."""
    import oracle
    oracle.build()
    X, y = data_np
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    k = min(wl.m, max(1, cores))
    rng = np.random.default_rng(3)
    members = list(range(k))
    kw = {}
    if emb is not None:   # the first k members' sizes and frequencies (stored member after member)
        n_f = wl.d_in * int(np.sum(emb["d_emb"][:k] - 1))
        kw = dict(d_emb=emb["d_emb"][:k], freq=emb["freq"][:n_f].astype(np.float64))
    pk = oracle.OraclePack(wl.d_in, wl.d_out, wl.task, hp["depth"][members], hp["width"][members],
                           hp["dropout"][members], hp["lr"][members], hp["wd"][members], seed=SEED_INIT,
                           member_id=members, **kw)
    if lr_muon is not None:
        pk.set_muon(np.asarray(lr_muon[:k], dtype=np.float64))
    steps = 0
    t0 = time.perf_counter()
    while True:
        if stacked:
            idx = np.stack([rng.choice(X.shape[0], B, replace=False) for _ in range(k)]).astype(np.int32)
        else:
            idx = rng.choice(X.shape[0], B, replace=False).astype(np.int32)
        pk.train_step(X, idx, y, steps)
        steps += 1
        el = time.perf_counter() - t0
        if el > budget_s or steps >= 50:
            break
    value = k * B * steps / el
    return {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"members 0..{k - 1} of {wl.m} (independent), {steps} full steps of batch {B}, {el:.1f} s"}


def emb_desc(emb):
    if emb is None:
        return "none (raw features)"
    return ("periodic (App. Feature Embeddings), d_emb UniformInt[8,32] step 4 (sampled %s), sigma "
            "LogUniform[1e-2,10]" % ",".join(str(int(x)) for x in emb["d_emb"]))


def run_reference(args, wl, rank):
    """Reference arm: the CPU fp64 oracle, as it stands, timed on the host
    cores (rank 0 only) over exactly W untimed and K timed steps.  Each step
    is a bounded sample of the workload: the first min(m, cores) members
    (independent of the others, one OpenMP thread each) on a batch whose rows
    are cut, when needed, so that the W + K steps fit in about
    --reference-seconds: a full-batch step and a one-row step calibrate the
    step time as a fixed cost (the optimizer pass over every parameter,
    operand copies) plus a cost per row."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    hp = sample_hparams(wl, seed=SEED_HP)
    B = wl.batch
    n = min(wl.n_train, 20000)
    d = make_data(wl, device="cpu", n_train=n, n_val=0)
    X, y = d["X_train"].numpy(), d["y_train"].numpy()
    emb = sample_emb(wl.m, wl.d_in, seed=SEED_HP + 200) if args.emb else None
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    k = min(wl.m, max(1, cores))
    members = list(range(k))
    kw = {}
    if emb is not None:
        n_f = wl.d_in * int(np.sum(emb["d_emb"][:k] - 1))
        kw = dict(d_emb=emb["d_emb"][:k], freq=emb["freq"][:n_f].astype(np.float64))
    pk = oracle.OraclePack(wl.d_in, wl.d_out, wl.task, hp["depth"][members], hp["width"][members],
                           hp["dropout"][members], hp["lr"][members], hp["wd"][members], seed=SEED_INIT,
                           member_id=members, **kw)
    if args.muon:
        pk.set_muon(muon_lrs(wl.m)[:k].astype(np.float64))
    rng = np.random.default_rng(3)

    def step(rows, s):
        if args.stacked:
            idx = np.stack([rng.choice(n, rows, replace=False) for _ in range(k)]).astype(np.int32)
        else:
            idx = rng.choice(n, rows, replace=False).astype(np.int32)
        pk.train_step(X, idx, y, s)

    t0 = time.perf_counter()
    step(B, 0)                                   # calibration steps (they count as warm-up)
    t_full = time.perf_counter() - t0
    t0 = time.perf_counter()
    step(1, 1)
    t_one = time.perf_counter() - t0
    per_row = max(t_full - t_one, 1e-9) / max(B - 1, 1)
    budget = float(args.reference_seconds) / max(1, args.steps + args.warmup)
    rows = B if t_full <= budget else max(1, min(B, int((budget - t_one) / per_row)))
    for s in range(2, args.warmup):
        step(rows, s)
    t0 = time.perf_counter()
    for s in range(args.steps):
        step(rows, args.warmup + s)
    el = time.perf_counter() - t0
    value = k * rows * args.steps / el
    sample = (f"members 0..{k - 1} of {wl.m} (independent, one thread each), {args.steps} timed steps of "
              f"{rows} row{'s' if rows != 1 else ''} each" + (f" (batch {B} cut to fit {args.reference_seconds:.0f} s; a full-batch step "
                                     f"took {t_full:.2f} s, a one-row step {t_one:.3f} s)" if rows < B
                                     else " (the full batch)") + f", {el:.1f} s")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": workload_desc(wl, B), "embeddings": emb_desc(emb),
                       "optimizer": "Muon (hidden weights) + AdamW" if args.muon else "AdamW",
                       "batches": "one per member (stacked)" if args.stacked else "one shared by all members"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": k, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="medium", choices=sorted(WORKLOADS))
    ap.add_argument("--precision", default="bf16", choices=["bf16", "fp32"])
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--members", type=int, default=0,
                    help="train only the first N members of the workload (profiling small cases)")
    ap.add_argument("--fuse-optimizer", action="store_true", help="AdamW inside the weight-gradient epilogue")
    ap.add_argument("--no-online", action="store_true", help="skip timing the online-ensemble epoch end")
    ap.add_argument("--online-score", default="loss", choices=["loss", "accuracy", "rmse", "auc"],
                    help="ensemble score of the timed online epoch end (auc: binary workloads)")
    ap.add_argument("--muon", action="store_true",
                    help="Muon for the hidden-layer weights (the paper's default optimizer), AdamW for the rest")
    ap.add_argument("--stacked", action="store_true",
                    help="a batch per member (idx [m, B], Sec. 3.6) instead of one batch shared by all members")
    ap.add_argument("--reference-seconds", type=float, default=120.0,
                    help="--impl reference: CPU seconds the W + K oracle steps are sized to")
    ap.add_argument("--emb", action="store_true",
                    help="periodic feature embeddings (App. Feature Embeddings), d_emb and sigma per member "
                         "from the paper's sampling space")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    wl = WORKLOADS[args.workload]
    if args.members > 0:
        import dataclasses
        wl = dataclasses.replace(wl, m=min(wl.m, args.members))

    if args.impl == "reference":
        run_reference(args, wl, rank)
        return

    import torch
    import torch.distributed as dist
    import paper_2607_05380_gb300 as tp

    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    tp.load_library()

    B = wl.batch
    hp = {k: v[:wl.m] for k, v in sample_hparams(WORKLOADS[args.workload], seed=SEED_HP).items()}
    d = make_data(wl, device=dev)
    X, y = d["X_train"], d["y_train"]
    n_train = X.shape[0]
    total = args.warmup + args.steps
    gen = torch.Generator(device=dev)
    gen.manual_seed(3)
    if args.stacked:   # [steps, m, B]: each member its own rows
        idx_all = torch.randint(0, n_train, (total, wl.m, B), generator=gen, device=dev)
    else:
        idx_all = torch.stack([torch.randperm(n_train, generator=gen, device=dev)[:B] for _ in range(total)])
    idx_all = idx_all.to(torch.int32).contiguous()

    stream = torch.cuda.current_stream()
    emb = sample_emb(wl.m, wl.d_in, seed=SEED_HP + 200) if args.emb else None
    pack = tp.Pack(wl.d_in, wl.d_out, wl.task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                   max_batch=B, seed=SEED_INIT, precision=args.precision, stream=stream,
                   fuse_optimizer=args.fuse_optimizer, d_emb=None if emb is None else emb["d_emb"],
                   freq=None if emb is None else emb["freq"])
    loss = torch.zeros(wl.m, dtype=torch.float32, device=dev)
    lr_muon = None
    if args.muon:
        lr_muon = muon_lrs(wl.m)
        pack.set_muon(lr_muon)

    for s in range(args.warmup):
        pack.train_step(X, idx_all[s], y, s, loss)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()

    gpu_id = getattr(torch.cuda.get_device_properties(dev), "uuid", None)
    gpu_id = f"GPU-{gpu_id}" if gpu_id is not None and not str(gpu_id).startswith("GPU-") else (gpu_id or local)
    l0 = pack.launch_count()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu_id) as clk:
        torch.cuda.synchronize()
        ev0.record(stream)
        for s in range(args.warmup, total):
            pack.train_step(X, idx_all[s], y, s, loss)
        ev1.record(stream)
        torch.cuda.synchronize()
    launches = pack.launch_count() - l0
    ms_total = ev0.elapsed_time(ev1)
    if world > 1:
        ms_total = max_over_ranks(ms_total, dist, dev)
        dist.barrier()
    ms_step = ms_total / args.steps
    value = job_rate(world, wl.m, B, args.steps, ms_total)
    lossv = loss.cpu().numpy()

    # per-kernel-family times over a second timed region (CUDA events on the pack's stream)
    pack.profile_enable(True)
    pack.profile_read(reset=True)
    n_prof = min(args.steps, 50)
    for s in range(n_prof):
        pack.train_step(X, idx_all[args.warmup + s], y, total + s, loss)
    prof = pack.profile_read(reset=True)
    pack.profile_enable(False)
    flops, n_params = work_per_step(wl, hp, B, emb)
    # the DRAM captures are of the default configuration (shared batch, AdamW, raw features)
    plain = args.members == 0 and not (args.emb or args.muon or args.stacked)
    pk = peaks()
    fam = {k: v for k, v in prof.items() if v[1] > 0}
    dominant = max(fam, key=lambda k: fam[k][0])
    shares = {k: round(v[0] / sum(x[0] for x in fam.values()), 4) for k, v in fam.items()}
    fwd_ms = prof["fwd"][0] / n_prof                              # per step
    bwd_ms = prof["bwd"][0] / n_prof
    adam_ms = prof["adamw"][0] / n_prof
    gemm_ms = fwd_ms + bwd_ms
    gemm = {"kernel": "k_tc_gemm (grouped fwd + dgrad + wgrad launches of one step)", "bound": "tensor",
            "achieved": flops / (gemm_ms / 1e3) / 1e12, "peak": pk["bf16_sus"], "unit": "TFLOP/s",
            "traffic": DRAM_TRAFFIC.get((args.workload, "k_tc_gemm")) if plain else None,
            "ms_per_step": gemm_ms, "peak_source": pk["source"] + " sustained bf16"}
    gemm["frac"] = gemm["achieved"] / gemm["peak"]
    if adam_ms > 0:   # AdamW as a separate pass (the default): 30 B per parameter
        mem = {"kernel": "k_adamw", "bound": "hbm", "achieved": 30.0 * n_params / (adam_ms / 1e3) / 1e9,
               "ms_per_step": adam_ms, "bytes_per_step": 30.0 * n_params}
    else:             # --fuse-optimizer: AdamW in the wgrad epilogue, 26 B per parameter
        mem = {"kernel": "k_tc_gemm backward launches (fused AdamW: read p, m, v; write p, m, v, bf16 p)",
               "bound": "hbm", "achieved": 26.0 * n_params / (bwd_ms / 1e3) / 1e9, "ms_per_step": bwd_ms,
               "bytes_per_step": 26.0 * n_params}
    mem.update({"peak": pk["hbm"], "unit": "GB/s", "peak_source": pk["source"] + " HBM copy",
                "traffic": DRAM_TRAFFIC.get((args.workload, "k_adamw")) if plain and adam_ms > 0 else None})
    mem["frac"] = mem["achieved"] / mem["peak"]
    roof = dict(gemm if gemm_ms >= adam_ms else mem)
    roof["other"] = mem if gemm_ms >= adam_ms else gemm
    roof["shares"] = shares
    if args.muon:   # the Newton-Schulz products: 5 x (4 r^2 c + 2 r^3) per matrix
        ns_flops = 0.0
        for i_, (L_, w_) in enumerate(zip(hp["depth"], hp["width"])):
            for l in range(int(L_)):
                cols = in0_of(wl, emb, i_) if l == 0 else int(w_)
                r_, c_ = min(int(w_), cols), max(int(w_), cols)
                ns_flops += 5 * (4.0 * r_ * r_ * c_ + 2.0 * r_ ** 3)
        muon_ms = prof["muon"][0] / n_prof
        roof["muon"] = {"kernels": "k_muon_* + k_tc_gemm Newton-Schulz launches", "ms_per_step": muon_ms,
                        "ns_flop_per_step": ns_flops, "achieved": ns_flops / (muon_ms / 1e3) / 1e12,
                        "unit": "TFLOP/s", "peak": pk["bf16_sus"], "frac": ns_flops / (muon_ms / 1e3) / 1e12 / pk["bf16_sus"]}

    # end to end through the public API with host buffers: per step the batch
    # rows and labels go host -> device (pinned), the member losses come back
    e2e = None
    if not args.no_e2e:
        Xh = X.cpu().pin_memory()
        yh = y.cpu().pin_memory()
        idx_h = idx_all.cpu()
        # per step the rows the step reads (stacked: m batches of B rows)
        xb_h = [Xh[idx_h[s].reshape(-1).long()].pin_memory() for s in range(min(total, 64))]
        yb_h = [yh[idx_h[s].reshape(-1).long()].pin_memory() for s in range(min(total, 64))]
        n_rows_step = xb_h[0].shape[0]
        ident = torch.arange(n_rows_step, dtype=torch.int32, device=dev)
        if args.stacked:
            ident = ident.view(wl.m, B)
        xb_d = torch.empty(n_rows_step, wl.d_in, dtype=torch.float32, device=dev)
        yb_d = torch.empty(n_rows_step, dtype=y.dtype, device=dev)
        loss_h = torch.empty(wl.m, dtype=torch.float32).pin_memory()
        n_e2e = min(args.steps, 64)
        for s in range(3):
            xb_d.copy_(xb_h[s], non_blocking=True)
            yb_d.copy_(yb_h[s], non_blocking=True)
            pack.train_step(xb_d, ident, yb_d, s, loss)
            loss_h.copy_(loss, non_blocking=True)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(n_e2e):
            xb_d.copy_(xb_h[s % len(xb_h)], non_blocking=True)
            yb_d.copy_(yb_h[s % len(yb_h)], non_blocking=True)
            pack.train_step(xb_d, ident, yb_d, 10_000 + s, loss)
            loss_h.copy_(loss, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        ms_e2e = max(e0.elapsed_time(e1), wall * 1000.0)
        e2e = {"value": world * wl.m * B * n_e2e / (ms_e2e / 1000.0), "unit": UNIT,
               "h2d_bytes_per_step": n_rows_step * (wl.d_in * 4 + 4), "d2h_bytes_per_step": wl.m * 4,
               "steps": n_e2e}

    online = None if args.no_online else time_online_epoch(tp, torch, pack, wl, hp, d, X, y, idx_all, stream, loss,
                                                           score=args.online_score, emb=emb)

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        n = min(n_train, 20000)
        data_np = (X[:n].cpu().numpy(), y[:n].cpu().numpy())
        cpu = cpu_baseline(wl, hp, data_np, B, budget_s=20.0, stacked=args.stacked, emb=emb, lr_muon=lr_muon)

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": args.precision, "data": "synthetic",
                "config": {"workload": workload_desc(wl, B), "precision": args.precision,
                           "params": n_params, "gemm_flop_per_step": flops,
                           "l2": "inputs larger than L2: each step streams ~%.2f GB of parameters and optimizer state"
                                 % (30.0 * n_params / 1e9),
                           "parallelism": "one independent pack per GPU" if world > 1 else "single GPU",
                           "batches": "one per member (stacked)" if args.stacked else "one shared by all members",
                           "optimizer": "Muon (hidden weights, lr LogUniform[1e-3, 1e-1]) + AdamW" if args.muon
                                        else "AdamW",
                           "embeddings": emb_desc(emb)},
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches, "online_epoch": online,
                "clocks": clk.summary(), "final_losses_mean": float(np.nanmean(lossv))}
        print(json.dumps(line), flush=True)
    pack.close()
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
