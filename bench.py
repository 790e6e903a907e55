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
# the current kernels (summaries in profiles/; the wide figures are captures of its
# first 4 members scaled to 16, the GEMM's by GEMM flops, AdamW's by parameters).
# A workload without a capture of the current kernel reports null.
DRAM_TRAFFIC = {
    ("medium", "k_adamw"): 607.7e6,
    ("wide", "k_tc_gemm"): 2.848e9,
    ("wide", "k_adamw"): 4.020e9,
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
    """SM clock, power and clock-event reasons of this GPU, sampled during the
    timed region: NVML through ctypes every 2 ms on a thread (the handle is
    found by the device's UUID, else its PCI bus id), else `nvidia-smi -lms 50`.
    The sampler takes its first sample before the region starts and keeps
    sampling until it ends, so even a region of a few milliseconds is
    covered."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown"}
    SMI_FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
                  "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
                  "clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid=None, pci=None, index=0):
        self.uuid, self.pci, self.index = uuid, pci, index
        self.samples = []          # (sm_mhz, max_mhz, reasons bitmask or names)
        self.source = None
        self._stop = threading.Event()
        self._thread = None
        self._proc = None

    def _nvml(self):
        import ctypes
        try:
            L = ctypes.CDLL("libnvidia-ml.so.1")
        except OSError:
            return None
        if L.nvmlInit_v2() != 0:
            return None
        h = ctypes.c_void_p()
        ok = False
        if self.uuid:
            ok = L.nvmlDeviceGetHandleByUUID(self.uuid.encode(), ctypes.byref(h)) == 0
        if not ok and self.pci:
            ok = L.nvmlDeviceGetHandleByPciBusId_v2(self.pci.encode(), ctypes.byref(h)) == 0
        if not ok:
            n = ctypes.c_uint(0)
            if L.nvmlDeviceGetCount_v2(ctypes.byref(n)) == 0 and n.value == 1:
                ok = L.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(h)) == 0
        if not ok:
            return None
        reasons_fn = getattr(L, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(L, "nvmlDeviceGetCurrentClocksThrottleReasons")
        return L, h, reasons_fn

    def _loop(self, L, h, reasons_fn):
        import ctypes
        clk, mx, rs = ctypes.c_uint(0), ctypes.c_uint(0), ctypes.c_ulonglong(0)
        while True:
            if (L.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and
                    L.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0 and
                    reasons_fn(h, ctypes.byref(rs)) == 0):
                self.samples.append((float(clk.value), float(mx.value), int(rs.value)))
            if self._stop.wait(0.002):
                break

    def __enter__(self):
        nv = None
        try:
            nv = self._nvml()
        except Exception:
            nv = None
        if nv is not None:
            self.source = "nvml"
            self._thread = threading.Thread(target=self._loop, args=nv, daemon=True)
            self._thread.start()
            t0 = time.time()
            while not self.samples and time.time() - t0 < 2.0:
                time.sleep(0.001)
            return self
        try:
            gid = self.uuid if self.uuid else str(self.index)
            self._proc = subprocess.Popen(["nvidia-smi", f"--id={gid}", f"--query-gpu={self.SMI_FIELDS}",
                                           "--format=csv,noheader,nounits", "-lms", "50"],
                                          stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.source = "nvidia-smi"
            time.sleep(1.0)            # its first lines come before the region starts
        except Exception:
            self._proc = None
        return self

    def __exit__(self, *a):
        if self._thread is not None:
            self._stop.set()
            self._thread.join(timeout=2)
        if self._proc is not None:
            time.sleep(0.1)
            self._proc.terminate()
            try:
                out, _ = self._proc.communicate(timeout=5)
            except Exception:
                self._proc.kill()
                out = ""
            names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
            for line in (out or "").strip().splitlines():
                f = [x.strip() for x in line.split(",")]
                if len(f) < 8:
                    continue
                try:
                    self.samples.append((float(f[0]), float(f[1]),
                                         [n for n, v in zip(names, f[4:8]) if v.lower().startswith("active")]))
                except ValueError:
                    continue

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "source": self.source}
        reasons = set()
        for _, _, r in self.samples:
            if isinstance(r, int):
                reasons.update(n for bit, n in self.REASONS.items() if r & bit)
            else:
                reasons.update(r)
        return {"sm_mhz": statistics.median(x[0] for x in self.samples),
                "sm_max_mhz": max(x[1] for x in self.samples), "samples": len(self.samples),
                "reasons": sorted(reasons), "source": self.source}


def device_ids(torch, dev):
    """(NVML UUID string, PCI bus id) of a torch device, where torch has them."""
    props = torch.cuda.get_device_properties(dev)
    uuid = getattr(props, "uuid", None)
    uuid = None if uuid is None else str(uuid)
    if uuid is not None and not uuid.startswith("GPU-"):
        uuid = "GPU-" + uuid
    pci = None
    if all(hasattr(props, k) for k in ("pci_domain_id", "pci_bus_id", "pci_device_id")):
        pci = "%08x:%02x:%02x.0" % (props.pci_domain_id, props.pci_bus_id, props.pci_device_id)
    return uuid, pci


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


def oracle_sample_pack(wl, hp, k, emb=None, lr_muon=None):
    """The oracle on the first k members of the workload (independent of the
    others), with their embeddings and Muon learning rates if any."""
    import oracle
    oracle.build()
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
    return pk


def oracle_rows(step, B, budget_s):
    """Rows per oracle step so that one step takes about budget_s: a step of
    min(B, 32) rows and a step of one row calibrate it as a fixed cost (the
    optimizer pass over every parameter, operand copies) plus a cost per row.
    Returns (rows, calibration note); the calibration steps count as warm-up."""
    r_cal = min(B, 32)
    t0 = time.perf_counter()
    step(r_cal)
    t_cal = time.perf_counter() - t0
    t0 = time.perf_counter()
    step(1)
    t_one = time.perf_counter() - t0
    per_row = max(t_cal - t_one, 1e-9) / max(r_cal - 1, 1)
    fixed = max(t_one - per_row, 0.0)
    rows = B if fixed + per_row * B <= budget_s else max(1, min(B, int((budget_s - fixed) / per_row)))
    note = (f"batch {B} cut to {rows} rows per step to fit the time budget (calibration: {r_cal} rows "
            f"{t_cal:.2f} s, 1 row {t_one:.3f} s)" if rows < B else f"the full batch of {B} rows")
    return rows, note


def cpu_baseline(wl, hp, data_np, B, budget_s=20.0, stacked=False, emb=None, lr_muon=None):
    """The oracle as it stands, on the host cores, on a bounded sample of the
    same workload: the first k members (independent of the others, one
    OpenMP thread each), timed over whole steps until about budget_s seconds
    of CPU work, each step's rows cut so that at least five steps fit
    (stacked: a batch per member; emb: the members' periodic embeddings;
    lr_muon: Muon for the hidden weights with these per-member learning
    rates)."""
    X, y = data_np
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    k = min(wl.m, max(1, cores))
    rng = np.random.default_rng(3)
    pk = oracle_sample_pack(wl, hp, k, emb, lr_muon)
    counter = [0]

    def step(rows):
        if stacked:
            idx = np.stack([rng.choice(X.shape[0], rows, replace=False) for _ in range(k)]).astype(np.int32)
        else:
            idx = rng.choice(X.shape[0], rows, replace=False).astype(np.int32)
        pk.train_step(X, idx, y, counter[0])
        counter[0] += 1

    rows, note = oracle_rows(step, B, budget_s / 5.0)
    steps = 0
    t0 = time.perf_counter()
    while True:
        step(rows)
        steps += 1
        el = time.perf_counter() - t0
        if el > budget_s or steps >= 50:
            break
    value = k * rows * steps / el
    return {"value": value, "unit": UNIT, "cores": k, "kind": "oracle",
            "sample": f"members 0..{k - 1} of {wl.m} (independent, one thread each), {steps} timed steps of "
                      f"{note}, {el:.1f} s"}


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
    --reference-seconds."""
    if rank != 0:
        return
    hp = sample_hparams(wl, seed=SEED_HP)
    hp = {k: v[:wl.m] for k, v in hp.items()}
    B = wl.batch
    n = min(wl.n_train, 20000)
    d = make_data(wl, device="cpu", n_train=n, n_val=0)
    X, y = d["X_train"].numpy(), d["y_train"].numpy()
    emb = sample_emb(wl.m, wl.d_in, seed=SEED_HP + 200) if args.emb else None
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    k = min(wl.m, max(1, cores))
    pk = oracle_sample_pack(wl, hp, k, emb, muon_lrs(wl.m) if args.muon else None)
    rng = np.random.default_rng(3)
    counter = [0]

    def step(rows):
        if args.stacked:
            idx = np.stack([rng.choice(n, rows, replace=False) for _ in range(k)]).astype(np.int32)
        else:
            idx = rng.choice(n, rows, replace=False).astype(np.int32)
        pk.train_step(X, idx, y, counter[0])
        counter[0] += 1

    rows, note = oracle_rows(step, B, float(args.reference_seconds) / max(1, args.steps + args.warmup))
    for _ in range(max(0, args.warmup - 2)):
        step(rows)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step(rows)
    el = time.perf_counter() - t0
    value = k * rows * args.steps / el
    sample = (f"members 0..{k - 1} of {wl.m} (independent, one thread each), {args.steps} timed steps of "
              f"{note}, {el:.1f} s")
    flops, n_params = work_per_step(wl, hp, B, emb)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": run_config(args, wl, B, n_params, flops, emb, world=1),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": k, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_config(args, wl, B, n_params, flops, emb, world):
    """The `config` object of a bench line (the same keys in both arms)."""
    return {"workload": workload_desc(wl, B), "params": n_params, "gemm_flop_per_step": flops,
            "l2": "inputs larger than L2: each step streams ~%.2f GB of parameters and optimizer state"
                  % (30.0 * n_params / 1e9),
            "parallelism": "one independent pack per GPU" if world > 1 else "single GPU",
            "batches": "one per member (stacked)" if args.stacked else "one shared by all members",
            "optimizer": "Muon (hidden weights, lr LogUniform[1e-3, 1e-1]) + AdamW" if args.muon else "AdamW",
            "embeddings": emb_desc(emb)}


def measure(args, tp, torch, dist, dev, name, steps, warmup, world, rank, headline):
    """Train the workload's pack for warmup + steps steps and time the last
    `steps` (CUDA events on the pack's stream, clocks sampled during the
    region), then the per-kernel-family profile.  headline: also the
    end-to-end leg, the online epoch end and the CPU baseline."""
    wl = WORKLOADS[name]
    if args.members > 0:
        import dataclasses
        wl = dataclasses.replace(wl, m=min(wl.m, args.members))
    B = wl.batch
    hp = {k: v[:wl.m] for k, v in sample_hparams(WORKLOADS[name], seed=SEED_HP).items()}
    d = make_data(wl, device=dev)
    X, y = d["X_train"], d["y_train"]
    n_train = X.shape[0]
    total = warmup + steps
    gen = torch.Generator(device=dev)
    gen.manual_seed(3)
    n_idx = min(total, 512)            # the batch index stream repeats after 512 steps
    if args.stacked:   # [steps, m, B]: each member its own rows
        idx_all = torch.randint(0, n_train, (n_idx, wl.m, B), generator=gen, device=dev)
    else:
        idx_all = torch.stack([torch.randperm(n_train, generator=gen, device=dev)[:B] for _ in range(n_idx)])
    idx_all = idx_all.to(torch.int32).contiguous()

    stream = torch.cuda.current_stream()
    emb = sample_emb(wl.m, wl.d_in, seed=SEED_HP + 200) if args.emb else None
    pack = tp.Pack(wl.d_in, wl.d_out, wl.task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                   max_batch=B, seed=SEED_INIT, precision=args.precision, stream=stream,
                   fuse_optimizer=args.fuse_optimizer, d_emb=None if emb is None else emb["d_emb"],
                   freq=None if emb is None else emb["freq"])
    if args.bias_path != "auto" and args.precision == "bf16":
        pack.debug_bias_path(1 if args.bias_path == "colsums" else 0)
    loss = torch.zeros(wl.m, dtype=torch.float32, device=dev)
    lr_muon = None
    if args.muon:
        lr_muon = muon_lrs(wl.m)
        pack.set_muon(lr_muon)

    for s in range(warmup):
        pack.train_step(X, idx_all[s % n_idx], y, s, loss)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()

    uuid, pci = device_ids(torch, dev)
    l0 = pack.launch_count()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(uuid, pci, dev.index or 0) as clk:
        torch.cuda.synchronize()
        ev0.record(stream)
        for s in range(warmup, total):
            pack.train_step(X, idx_all[s % n_idx], y, s, loss)
        ev1.record(stream)
        torch.cuda.synchronize()
    launches = pack.launch_count() - l0
    ms_total = ev0.elapsed_time(ev1)
    if world > 1:
        ms_total = max_over_ranks(ms_total, dist, dev)
        dist.barrier()
    ms_step = ms_total / steps
    value = job_rate(world, wl.m, B, steps, ms_total)
    lossv = loss.cpu().numpy()

    # per-kernel-family times over a second timed region (CUDA events on the pack's stream)
    pack.profile_enable(True)
    pack.profile_read(reset=True)
    n_prof = min(steps, 50)
    for s in range(n_prof):
        pack.train_step(X, idx_all[(warmup + s) % n_idx], y, total + s, loss)
    prof = pack.profile_read(reset=True)
    pack.profile_enable(False)
    flops, n_params = work_per_step(wl, hp, B, emb)
    # the DRAM captures are of the default configuration (shared batch, AdamW, raw features)
    plain = args.members == 0 and not (args.emb or args.muon or args.stacked)
    pk = peaks()
    # a region well under a second runs at the burst clocks; a long one under the power cap
    burst = ms_total < 1000.0
    tensor_peak = pk["bf16"] if burst else pk["bf16_sus"]
    peak_note = pk["source"] + (" bf16 burst (timed region %.0f ms < 1 s)" % ms_total if burst
                                else " bf16 sustained (timed region %.1f s)" % (ms_total / 1e3))
    fam = {k: v for k, v in prof.items() if v[1] > 0}
    shares = {k: round(v[0] / sum(x[0] for x in fam.values()), 4) for k, v in fam.items()}
    fwd_ms = prof["fwd"][0] / n_prof                              # per step
    bwd_ms = prof["bwd"][0] / n_prof
    adam_ms = prof["adamw"][0] / n_prof
    gemm_ms = fwd_ms + bwd_ms
    gemm = {"kernel": "k_tc_gemm (grouped fwd + dgrad + wgrad launches of one step)", "bound": "tensor",
            "achieved": flops / (gemm_ms / 1e3) / 1e12, "peak": tensor_peak, "unit": "TFLOP/s",
            "traffic": DRAM_TRAFFIC.get((name, "k_tc_gemm")) if plain else None,
            "ms_per_step": gemm_ms, "peak_source": peak_note}
    gemm["frac"] = gemm["achieved"] / gemm["peak"]
    n_adam = n_params
    if args.muon:     # AdamW keeps the biases and the head; Muon the hidden weight matrices
        n_adam -= sum(in0_of(wl, emb, i_) * int(w_) + (int(L_) - 1) * int(w_) ** 2
                      for i_, (L_, w_) in enumerate(zip(hp["depth"], hp["width"])))
    if adam_ms > 0:   # AdamW as a separate pass (the default): 30 B per parameter
        mem = {"kernel": "k_adamw", "bound": "hbm", "achieved": 30.0 * n_adam / (adam_ms / 1e3) / 1e9,
               "ms_per_step": adam_ms, "bytes_per_step": 30.0 * n_adam}
    else:             # --fuse-optimizer: AdamW in the wgrad epilogue, 26 B per parameter
        mem = {"kernel": "k_tc_gemm backward launches (fused AdamW: read p, m, v; write p, m, v, bf16 p)",
               "bound": "hbm", "achieved": 26.0 * n_params / (bwd_ms / 1e3) / 1e9, "ms_per_step": bwd_ms,
               "bytes_per_step": 26.0 * n_params}
    mem.update({"peak": pk["hbm"], "unit": "GB/s", "peak_source": pk["source"] + " HBM copy",
                "traffic": DRAM_TRAFFIC.get((name, "k_adamw")) if plain and adam_ms > 0 else None})
    mem["frac"] = mem["achieved"] / mem["peak"]
    roof = dict(gemm if gemm_ms >= adam_ms else mem)
    roof["other"] = mem if gemm_ms >= adam_ms else gemm
    roof["shares"] = shares
    roof["step_tflops"] = flops / (ms_step / 1e3) / 1e12
    roof["step_frac"] = roof["step_tflops"] / tensor_peak
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
                        "unit": "TFLOP/s", "peak": tensor_peak, "frac": ns_flops / (muon_ms / 1e3) / 1e12 / tensor_peak}
    out = {"wl": wl, "hp": hp, "B": B, "value": value, "ms_step": ms_step, "flops": flops, "n_params": n_params,
           "roof": roof, "launches": launches, "clocks": clk.summary(), "loss": float(np.nanmean(lossv)),
           "emb": emb}
    if not headline:
        pack.close()
        return out

    # end to end through the public API with host buffers: per step the batch
    # rows and labels go host -> device (pinned), the member losses come back
    e2e = None
    if not args.no_e2e:
        Xh = X.cpu().pin_memory()
        yh = y.cpu().pin_memory()
        idx_h = idx_all.cpu()
        # per step the rows the step reads (stacked: m batches of B rows)
        xb_h = [Xh[idx_h[s].reshape(-1).long()].pin_memory() for s in range(min(n_idx, 64))]
        yb_h = [yh[idx_h[s].reshape(-1).long()].pin_memory() for s in range(min(n_idx, 64))]
        n_rows_step = xb_h[0].shape[0]
        ident = torch.arange(n_rows_step, dtype=torch.int32, device=dev)
        if args.stacked:
            ident = ident.view(wl.m, B)
        # a double-buffered loader: step s + 1's rows and labels are copied on
        # a copy stream into the other device buffer while step s runs
        xb_d = [torch.empty(n_rows_step, wl.d_in, dtype=torch.float32, device=dev) for _ in range(2)]
        yb_d = [torch.empty(n_rows_step, dtype=y.dtype, device=dev) for _ in range(2)]
        loss_h = torch.empty(wl.m, dtype=torch.float32).pin_memory()
        copy_stream = torch.cuda.Stream(device=dev)
        ev_copied = [torch.cuda.Event() for _ in range(2)]
        ev_free = [torch.cuda.Event() for _ in range(2)]

        def issue_copy(s):
            b = s % 2
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(ev_free[b])  # the step that last read buffer b has run
                xb_d[b].copy_(xb_h[s % len(xb_h)], non_blocking=True)
                yb_d[b].copy_(yb_h[s % len(yb_h)], non_blocking=True)
                ev_copied[b].record(copy_stream)

        def run_steps(n, step0):
            issue_copy(0)
            for s in range(n):
                if s + 1 < n:
                    issue_copy(s + 1)
                stream.wait_event(ev_copied[s % 2])
                pack.train_step(xb_d[s % 2], ident, yb_d[s % 2], step0 + s, loss)
                ev_free[s % 2].record(stream)
                loss_h.copy_(loss, non_blocking=True)

        for b in range(2):
            ev_free[b].record(stream)
        n_e2e = min(steps, 64)
        run_steps(3, 0)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        copy_stream.wait_event(e0)  # every copy lies inside the timed region
        run_steps(n_e2e, 10_000)
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        ms_e2e = max(e0.elapsed_time(e1), wall * 1000.0)
        e2e = {"value": world * wl.m * B * n_e2e / (ms_e2e / 1000.0), "unit": UNIT,
               "h2d_bytes_per_step": n_rows_step * (wl.d_in * 4 + 4), "d2h_bytes_per_step": wl.m * 4,
               "steps": n_e2e,
               "note": "a host loader's batches: each step's rows and labels, gathered on the host before the "
                       "timed region (%d distinct batches, cycled), are copied from pinned memory on a copy "
                       "stream into one of two device buffers while the previous step runs; the step runs on "
                       "identity indices, the member losses come back" % len(xb_h)}
    out["e2e"] = e2e
    out["online"] = None if args.no_online else time_online_epoch(tp, torch, pack, wl, hp, d, X, y, idx_all, stream,
                                                                  loss, score=args.online_score, emb=emb)
    out["cpu"] = None
    if rank == 0 and not args.no_cpu_baseline:
        n = min(n_train, 20000)
        data_np = (X[:n].cpu().numpy(), y[:n].cpu().numpy())
        out["cpu"] = cpu_baseline(wl, hp, data_np, B, budget_s=20.0, stacked=args.stacked, emb=emb, lr_muon=lr_muon)
    pack.close()
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default="wide", choices=sorted(WORKLOADS))
    ap.add_argument("--also", default="medium,large,narrow",
                    help="further workloads timed in the same run and reported under `workloads` ('' for none)")
    ap.add_argument("--also-steps", type=int, default=100, help="timed steps of each further workload")
    ap.add_argument("--precision", default="bf16", choices=["bf16", "fp32"])
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--members", type=int, default=0,
                    help="train only the first N members of the workload (profiling small cases)")
    ap.add_argument("--fuse-optimizer", action="store_true", help="AdamW inside the weight-gradient epilogue")
    ap.add_argument("--bias-path", default="auto", choices=["auto", "colsums", "column"],
                    help="bf16: hidden-layer bias gradients from dZ column sums (where the input width is a "
                         "multiple of 256) or from a bias column; auto = the pack's own choice")
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

    head = measure(args, tp, torch, dist, dev, args.workload, args.steps, args.warmup, world, rank, True)
    others = {}
    for name in [n.strip() for n in args.also.split(",") if n.strip()]:
        if name == args.workload or name not in WORKLOADS:
            continue
        torch.cuda.empty_cache()
        o = measure(args, tp, torch, dist, dev, name, max(args.also_steps, 20), max(args.warmup, 5), world, rank,
                    False)
        r = o["roof"]
        g = r if r["bound"] == "tensor" else r["other"]
        a = r["other"] if r["bound"] == "tensor" else r
        others[name] = {"workload": workload_desc(o["wl"], o["B"]), "value": o["value"], "unit": UNIT,
                        "ms_per_step": o["ms_step"], "steps": max(args.also_steps, 20),
                        "gemm_tflops": g["achieved"], "gemm_frac": g["frac"], "gemm_ms_per_step": g["ms_per_step"],
                        "adamw_gbs": a["achieved"], "adamw_frac": a["achieved"] / a["peak"],
                        "adamw_ms_per_step": a["ms_per_step"], "step_frac": r["step_frac"], "shares": r["shares"],
                        "tensor_peak": g["peak"], "clocks": o["clocks"]}

    if rank == 0:
        line = {"metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": head["ms_step"], "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": args.precision, "data": "synthetic",
                "config": run_config(args, head["wl"], head["B"], head["n_params"], head["flops"], head["emb"], world),
                "roofline": head["roof"], "cpu_baseline": head["cpu"], "e2e": head["e2e"],
                "gpu_launches": head["launches"], "online_epoch": head["online"], "clocks": head["clocks"],
                "final_losses_mean": head["loss"], "workloads": others}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
