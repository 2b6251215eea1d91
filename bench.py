#!/usr/bin/env python
"""Benchmark of the decoupled off-policy correction hot path on GB300.

One step = the whole path over one batch: log pi_old of the sampled tokens
over the old logits, the decoupled loss forward + dlogits on the current
logits (by default both in the one-launch occ_decoupled_loss_fused; with
--loss-path two-call as occ_token_logprob + occ_decoupled_loss_fwd_bwd), and
the PPO-EWMA update of 7.6e9 float32 proximal parameters, auto-reset fed by
the loss statistics.  Workload: T=65536 tokens packed from 128
sequences, V=151936, bf16 logits (the agentic batch), seeded synthetic data.
Inputs (40 GB of logits, 61 GB of EWMA buffers) are far larger than L2, so no
flush is needed between steps.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Prints one JSON line (rank 0).  Under torchrun every rank runs a replica of
the workload on its own batch (weak scaling); the only exchange is the
all-reduce of the loss statistics before the EWMA reset decision.
"""

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "correction-loss tokens/s fwd+bwd at V=151936; HBM GB/s vs peak"
WORKLOAD = "agentic_bf16_v151936"
EWMA_BETA = 0.99
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0   # HBM3e spec-sheet figure, for context next to the measured peak


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--ewma-n", type=int, default=7_600_000_000)
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-graph", action="store_true",
                    help="skip timing the step replayed from a captured CUDA graph")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--tau", type=float, default=0.5)
    ap.add_argument("--tokens", type=int, default=None, help="resize T (profiling runs only)")
    ap.add_argument("--vocab", type=int, default=None,
                    help="resize V (profiling runs only; an odd V puts the bf16 rows off 16-byte "
                         "boundaries, which the peeled kernels take)")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="loss batch (default: the agentic batch the metric is quoted on; the "
                         "others are for breakdowns only)")
    ap.add_argument("--ewma-variants", action="store_true",
                    help="instead of the step, time the bf16 and host-resident EWMA buffers")
    ap.add_argument("--loss-path", default="fused", choices=["fused", "two-call"],
                    help="fused: one launch reads old and current logits (occ_decoupled_loss_fused); "
                         "two-call: occ_token_logprob then occ_decoupled_loss_fwd_bwd")
    ap.add_argument("--write-traffic", nargs=4, metavar=("CSVS", "T", "N_VALID", "N_PARAMS"),
                    help="no GPU: turn ncu CSVs of dram__bytes_{read,write}.sum (comma-separated, "
                         "one capture per kernel, of a run of this script on --workload with T "
                         "tokens, N_VALID of them valid, and N_PARAMS EWMA parameters) into "
                         "profiles/traffic_per_unit.json")
    return ap.parse_args()


# ----------------------------------------------------------------- helpers

def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "of measured"
    except Exception:
        return FALLBACK_HBM_GBS, "of fallback"


class ClockSampler:
    """nvidia-smi clock/throttle sampling while the timed region runs."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu_id), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except FileNotFoundError:
            self.proc = None
            return
        t0 = time.time()
        while time.time() - t0 < 5 and os.path.getsize(self.path) == 0:
            time.sleep(0.05)

    def stop(self, t_begin, t_end):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait(timeout=10)
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                    rows.append((ts, float(parts[1]), float(parts[2]), parts[3], *parts[4:9]))
                except ValueError:
                    continue
        os.unlink(self.path)
        inside = [r for r in rows if t_begin - 1 <= r[0] <= t_end + 1] or rows
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = sorted(r[1] for r in inside)
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in inside:
            for name, val in zip(names, r[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[2] for r in inside),
                "samples": len(inside), "reasons": sorted(reasons)}


KERNEL_SOURCES = {
    "k1_token_logprob": ("occ_logprob.cu", "occ_common.cuh"),
    "k2_decoupled_loss_fwd_bwd": ("occ_loss.cu", "occ_loss_common.cuh", "occ_common.cuh"),
    "k12_decoupled_loss_fused": ("occ_fused.cu", "occ_fused_common.cuh", "occ_loss_common.cuh",
                                 "occ_common.cuh"),
    "k3_ewma_update": ("occ_ewma.cu", "occ_common.cuh"),
}


_CODE_TOKENS = re.compile(r'"(?:\\.|[^"\\\n])*"|//[^\n]*|/\*.*?\*/', re.S)


def _code_only(src):
    """C++/CUDA source with comments removed and whitespace runs collapsed
    (string literals kept), so that a comment edit keeps a capture valid."""
    src = _CODE_TOKENS.sub(lambda m: m.group(0) if m.group(0).startswith('"') else " ", src)
    return " ".join(src.split())


def kernel_source_hash(name):
    """Hash of the code a kernel is built from, comments and layout aside (its
    traffic capture stays valid while that code is unchanged)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2605_12070_gb300", "csrc")
    for f in KERNEL_SOURCES[name]:
        with open(os.path.join(csrc, f)) as fh:
            h.update(f.encode() + _code_only(fh.read()).encode())
    return h.hexdigest()[:16]


TRAFFIC_JSON = os.path.join(ROOT, "profiles", "traffic_per_unit.json")


def ncu_traffic(workload, V, path=TRAFFIC_JSON):
    """Per-unit DRAM bytes from the committed ncu summary
    (profiles/traffic_per_unit.json) for the kernels whose sources have not
    changed since the capture, when the loss batch is the captured one (its
    recipe and V: per-token bytes depend on both; the EWMA's per-parameter
    bytes do not)."""
    try:
        with open(path) as f:
            d = json.load(f)
    except Exception:
        return {}
    same_batch = d.get("workload") == workload and d.get("V") == V
    return {k: v for k, v in d.get("kernels", {}).items()
            if k in KERNEL_SOURCES and v.get("source_hash") == kernel_source_hash(k)
            and (same_batch or k == "k3_ewma_update")}


# kernel-name prefix in an ncu launch list -> KERNEL_SOURCES key
_TRAFFIC_KERNELS = {"k1_logprob_vec": "k1_token_logprob", "k2_loss_l2": "k2_decoupled_loss_fwd_bwd",
                    "k2_fused_l2": "k12_decoupled_loss_fused", "k3_ewma_vec": "k3_ewma_update"}


def write_traffic(csv_path, workload, V, T, n_valid, n_params, command, path=TRAFFIC_JSON):
    """Reads one or more ncu CSVs (comma-separated paths; one capture per
    kernel), averages each kernel's DRAM bytes over its captured launches and stores
    them per unit (tokens, valid tokens, parameters) with the kernel's source
    hash in profiles/traffic_per_unit.json."""
    import csv
    rows = []
    for one in csv_path.split(","):
        with open(one) as f:
            rows += list(csv.DictReader([ln for ln in f if ln.startswith('"')]))
    acc = {}
    for r in rows:
        name = r["Kernel Name"].split("(")[0].replace("void ", "").strip()
        key = next((k for p, k in _TRAFFIC_KERNELS.items() if name.startswith(p)), None)
        metric = r["Metric Name"]
        if key and metric in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
            scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9}[r.get("Metric Unit",
                                                                              "byte")]
            v = float(r["Metric Value"].replace(",", "")) * scale
            acc.setdefault(key, {}).setdefault(metric, []).append(v)
    kernels = {}
    for key, d in acc.items():
        rd = sum(d["dram__bytes_read.sum"]) / len(d["dram__bytes_read.sum"])
        wr = sum(d["dram__bytes_write.sum"]) / len(d["dram__bytes_write.sum"])
        if key == "k1_token_logprob":
            e = {"read_per_token": rd / T, "write_per_token": wr / T}
        elif key == "k3_ewma_update":
            e = {"read_per_param": rd / n_params, "write_per_param": wr / n_params}
        else:
            e = {"read_per_valid_token": rd / n_valid, "write_per_token": wr / T}
        e["launches"] = len(d["dram__bytes_read.sum"])
        e["source_hash"] = kernel_source_hash(key)
        kernels[key] = e
    # entries of kernels left out of this capture stay while their code is unchanged
    try:
        with open(path) as f:
            old = json.load(f)
        if old.get("workload") == workload and old.get("V") == V:
            for key, e in old.get("kernels", {}).items():
                if key not in kernels and key in KERNEL_SOURCES \
                        and e.get("source_hash") == kernel_source_hash(key):
                    kernels[key] = e
    except (OSError, ValueError):
        pass
    kernels = dict(sorted(kernels.items()))
    out = {
        "what": (f"DRAM bytes per unit from ncu captures, one kernel per capture "
                 f"(dram__bytes_read.sum, dram__bytes_write.sum), of a run with T={T} tokens "
                 f"({n_valid} valid) and "
                 f"{n_params} EWMA parameters, averaged over the captured launches of each "
                 f"kernel; bench.py scales them to its workload by the units processed (valid "
                 f"tokens for the logits reads of the loss kernels, tokens for everything else, "
                 f"parameters for the EWMA). Writes are slightly under-counted: a single launch "
                 f"leaves up to ~60 MB of dirty lines in L2. Each entry is valid while its "
                 f"kernel's code (comments and layout aside) hashes to source_hash."),
        "command": command,
        "workload": workload,
        "V": V,
        "kernels": kernels,
    }
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    return out


def traffic_bytes(tr, name, T, n_valid, n_params):
    """DRAM bytes of one launch, scaled from the per-unit capture."""
    k = tr.get(name)
    if k is None:
        return None
    if name == "k1_token_logprob":
        return round(T * (k["read_per_token"] + k["write_per_token"]))
    if name in ("k2_decoupled_loss_fwd_bwd", "k12_decoupled_loss_fused"):
        return round(n_valid * k["read_per_valid_token"] + T * k["write_per_token"])
    return round(n_params * (k["read_per_param"] + k["write_per_param"]))


# ----------------------------------------------------------------- the oracle arm

_EWMA_SAMPLE = {}


def _ewma_sample(n):
    """Host EWMA buffers of n elements (drawn once per size; theta ~ N(0, 0.02^2),
    theta_prox = theta + N(0, 1e-4^2), like the device buffers)."""
    if n not in _EWMA_SAMPLE:
        import torch
        g = torch.Generator().manual_seed(0)
        th = (0.02 * torch.randn(n, generator=g)).numpy()
        _EWMA_SAMPLE.clear()
        _EWMA_SAMPLE[n] = (th, th + 1e-4 * torch.randn(n, generator=g).numpy())
    return _EWMA_SAMPLE[n]


def oracle_sample_times(batch, rows, n_params, threads):
    """Times the float64 oracle on `rows` tokens and `n_params` EWMA elements.
    Inputs are copied to the host before the clock starts."""
    import numpy as np
    import torch

    import oracle
    from oracle.rows import map_row_chunks
    rows = np.asarray(rows)
    it = torch.as_tensor(rows, device=batch.z_theta.device)
    zt = batch.z_theta[it].cpu()
    zo = batch.z_old[it].cpu()
    ids = batch.ids.cpu().numpy().astype(np.int64)
    mask = None if batch.mask is None else batch.mask.cpu().numpy()
    N = int(mask.sum()) if mask is not None else batch.T
    lmu = batch.logp_mu.cpu().numpy()[rows]
    adv = batch.adv.cpu().numpy()[rows]
    m = None if mask is None else mask[rows]
    p = oracle.LossParams(**batch.thresholds())
    th, tp = _ewma_sample(n_params)
    pos = {int(r): k for k, r in enumerate(rows)}

    def one(chunk):
        k = np.array([pos[int(r)] for r in chunk])
        z_old = zo[k].to(torch.float64).numpy()
        z = zt[k].to(torch.float64).numpy()
        lo, _ = oracle.token_logprob(z_old, ids[chunk])
        lt, lse = oracle.token_logprob(z, ids[chunk])
        terms = oracle.token_terms(lt, lo.astype(np.float32), lmu[k], adv[k],
                                   None if m is None else m[k], p,
                                   id_ok=(ids[chunk] >= 0), N=N)
        dz = oracle.softmax_grad_rows(z, ids[chunk], lse, terms["g"])
        return float(terms["loss_sum"]) + float(dz[0, 0])

    t0 = time.perf_counter()
    map_row_chunks(one, rows, chunk=max(1, len(rows) // threads), threads=threads)
    t_rows = time.perf_counter() - t0

    def ewma_part(ix):
        sl = slice(int(ix[0]), int(ix[-1]) + 1)
        oracle.ewma_update(tp[sl], th[sl], EWMA_BETA, oracle.EwmaState(w=1 / (1 - EWMA_BETA)))
        return 0

    t0 = time.perf_counter()
    map_row_chunks(ewma_part, np.arange(n_params), chunk=max(1, n_params // threads),
                   threads=threads)
    t_par = time.perf_counter() - t0
    return t_rows, t_par


# One oracle step: REF_SAMPLE_TOKENS tokens drawn from the batch and the same
# share of the EWMA parameters (n_params x tokens / T), so that the sample has
# the full step's mix of loss and EWMA work.  Shared by the cpu_baseline leg
# and the reference arm (smaller calls time the thread pool and numpy's
# per-array overhead instead of the oracle).
REF_SAMPLE_TOKENS = 512


def sample_params(T, n_params_full, tokens=REF_SAMPLE_TOKENS):
    """EWMA parameters that go with `tokens` of a T-token step."""
    return max(1, round(n_params_full * tokens / T))


def oracle_steps(batch, n_params_full, rng, steps=None, seconds=None):
    """Runs oracle sample steps (a fixed number, or until `seconds` of work) and
    returns (tokens per step, params per step, list of step times in s)."""
    import numpy as np

    from oracle.rows import host_cores
    threads = host_cores()
    S = min(REF_SAMPLE_TOKENS, batch.T)
    P = sample_params(batch.T, n_params_full, S)
    times = []
    while (steps is not None and len(times) < steps) or \
            (steps is None and sum(times) < seconds):
        rows = np.sort(rng.choice(batch.T, size=S, replace=False))
        tr, tp = oracle_sample_times(batch, rows, P, threads)
        times.append(tr + tp)
    return S, P, times, threads


def cpu_baseline(batch, n_params_full, seconds):
    """Times the oracle, as it stands, on sample steps of the workload for
    about `seconds` of work."""
    import numpy as np
    S, P, times, threads = oracle_steps(batch, n_params_full, np.random.default_rng(0),
                                        seconds=seconds)
    t = sum(times)
    return {
        "value": round(S * len(times) / t, 3), "unit": "tokens/s", "cores": threads,
        "kind": "oracle",
        "sample": (f"{len(times)} oracle steps of {S} tokens drawn from the T={batch.T}, "
                   f"V={batch.V} batch (log pi_old, loss, dlogits) and {P} EWMA parameters "
                   f"(the step's parameters-per-token), {t:.1f} s in all, on {threads} threads"),
        "seconds": round(t, 2),
    }


# ----------------------------------------------------------------- main

# The small case the traffic captures run on, and the captures themselves:
# one kernel per ncu run (an exact kernel name, two launches after the first),
# each after the same command has exited 0 without ncu.
TRAFFIC_CASE = ("python bench.py --tokens 4096 --ewma-n 200000000 --steps 2 --warmup 1 --no-e2e "
                "--no-cpu-baseline --no-graph")
TRAFFIC_KERNELS = ("k2_fused_l2", "k1_logprob_vec", "k2_loss_l2", "k3_ewma_vec")
TRAFFIC_COMMAND = (
    TRAFFIC_CASE + " > plain_small.log && for k in " + " ".join(TRAFFIC_KERNELS) + "; do "
    "ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum,gpu__time_duration.sum "
    "--clock-control none -k regex:^$k -s 1 -c 2 --csv --log-file traffic_$k.csv " + TRAFFIC_CASE +
    " > /dev/null || break; done; then python bench.py --write-traffic "
    + ",".join(f"traffic_{k}.csv" for k in TRAFFIC_KERNELS) + " 4096 <valid tokens> 200000000")


def main():
    args = parse_args()
    if args.write_traffic:
        csv_path, T, n_valid, n_params = args.write_traffic
        from paper_2605_12070_gb300.workloads import WORKLOADS
        out = write_traffic(csv_path, args.workload, WORKLOADS[args.workload]["V"], int(T),
                            int(n_valid), int(n_params), TRAFFIC_COMMAND)
        print(json.dumps(out["kernels"], indent=1))
        return
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        # The oracle arm: rank 0 alone, and nothing of the CUDA library (no
        # build, no libocc.so); the seeded generator only draws the batch.
        if rank != 0:
            return
        from paper_2605_12070_gb300.workloads import make_loss_batch
        dev = torch.device(f"cuda:{local}" if torch.cuda.is_available() else "cpu")
        if dev.type == "cuda":
            torch.cuda.set_device(dev)
        batch = make_loss_batch(args.workload, T=args.tokens, V=args.vocab, seed=0, device=dev)
        run_reference(args, batch, world)
        return
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)

    import __graft_entry__
    __graft_entry__.build()
    from paper_2605_12070_gb300 import dp, occ
    from paper_2605_12070_gb300.workloads import make_ewma_buffers, make_loss_batch

    batch = make_loss_batch(args.workload, T=args.tokens, V=args.vocab, seed=rank, device=dev)
    T, V = batch.T, batch.V
    n_valid = T if batch.mask is None else int(batch.mask.sum().item())

    if args.ewma_variants:
        del batch
        run_ewma_variants(args, dev)
        return

    theta, theta_prox = make_ewma_buffers(args.ewma_n, seed=rank, device=dev)
    state = occ.new_ewma_state(dev, w0=1.0 / (1.0 - EWMA_BETA))
    lp_old = torch.empty(T, dtype=torch.float32, device=dev)
    dlogits = torch.empty((T, V), dtype=batch.z_theta.dtype, device=dev)
    logp = torch.empty(T, dtype=torch.float32, device=dev)
    flags = torch.empty(T, dtype=torch.uint8, device=dev)
    stats = occ.new_loss_stats(dev)
    ws = occ.new_workspace(T, V, dev)
    denom = dp.global_token_count(n_valid) if world > 1 else 0
    stream = torch.cuda.current_stream(dev)

    def loss_two_call(ev=None):
        if ev is not None:
            ev[0].record(stream)
        occ.occ_token_logprob(batch.z_old, batch.ids, logp_out=lp_old)
        if ev is not None:
            ev[1].record(stream)
        occ.occ_decoupled_loss_fwd_bwd(batch.z_theta, batch.ids, lp_old, batch.logp_mu, batch.adv,
                                       batch.mask, **batch.thresholds(), denom=denom,
                                       dlogits=dlogits, logp_out=logp, flags_out=flags,
                                       stats=stats, workspace=ws)

    def loss_fused(ev=None):
        if ev is not None:
            ev[0].record(stream)
            ev[1].record(stream)
        occ.occ_decoupled_loss_fused(batch.z_theta, batch.z_old, batch.ids, batch.logp_mu,
                                     batch.adv, batch.mask, **batch.thresholds(), denom=denom,
                                     dlogits=dlogits, logp_out=logp, logp_old_out=lp_old,
                                     flags_out=flags, stats=stats, workspace=ws)

    loss = loss_fused if args.loss_path == "fused" else loss_two_call

    def step(ev=None, loss_fn=None):
        (loss_fn or loss)(ev)
        if world > 1:
            dp.allreduce_loss_stats(stats)
        if ev is not None:
            ev[2].record(stream)
        occ.occ_ewma_update(theta_prox, theta, EWMA_BETA, state, stats=stats, tau=args.tau)
        if ev is not None:
            ev[3].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()

    gpu_id = 0
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid).replace("GPU-", "")
    except Exception:
        gpu_id = local
    resets_before = occ.decode_ewma_state(state).n_resets
    clocks = ClockSampler(gpu_id)
    clocks.start()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    t_begin = time.time()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for k in range(args.steps):
        step(evs[k])
    end.record(stream)
    torch.cuda.synchronize()
    t_end = time.time()
    if world > 1:
        dist.barrier()
    clk = clocks.stop(t_begin, t_end)
    elapsed = start.elapsed_time(end) / 1e3
    if world > 1:
        t = torch.tensor([elapsed], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        elapsed = float(t.item())
    k1 = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps / 1e3
    k2 = sum(e[1].elapsed_time(e[2]) for e in evs) / args.steps / 1e3
    k3 = sum(e[2].elapsed_time(e[3]) for e in evs) / args.steps / 1e3
    ms_step = elapsed / args.steps * 1e3
    resets = occ.decode_ewma_state(state).n_resets - resets_before

    # the other loss path, timed the same way on the same inputs (breakdown only)
    alt_fn = loss_two_call if args.loss_path == "fused" else loss_fused
    for _ in range(2):
        step(loss_fn=alt_fn)
    aevs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(10)]
    for k in range(10):
        step(aevs[k], loss_fn=alt_fn)
    torch.cuda.synchronize()
    alt_k1 = sum(e[0].elapsed_time(e[1]) for e in aevs) / 10 / 1e3
    alt_k2 = sum(e[1].elapsed_time(e[2]) for e in aevs) / 10 / 1e3

    # the same step captured once as a CUDA graph and replayed (no host work per step)
    graph = None
    if world == 1 and not args.no_graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            step()
        for _ in range(2):
            g.replay()
        gs, ge = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        gs.record(stream)
        for _ in range(args.steps):
            g.replay()
        ge.record(stream)
        torch.cuda.synchronize()
        gsec = gs.elapsed_time(ge) / 1e3 / args.steps
        graph = {"ms_per_step": round(gsec * 1e3, 4), "tokens_per_s": round(T / gsec, 1),
                 "steps": args.steps,
                 "launches_per_replay": 5 if args.loss_path == "fused" else 6}

    peak, peak_kind = measured_peak()
    traffic = ncu_traffic(args.workload, V)
    es = batch.z_theta.element_size()
    bytes_k1 = T * V * es + T * 8
    bytes_k2 = n_valid * V * es + T * V * es + T * 37
    bytes_fused = 2 * n_valid * V * es + T * V * es + T * 41
    # a regular update reads theta_prox and theta and writes theta_prox; a reset copies theta
    bytes_k3 = args.ewma_n * (12 * (args.steps - resets) + 8 * resets) // args.steps
    st_last = occ.decode_loss_stats(stats)
    if args.loss_path == "fused":
        kern = {"k12_decoupled_loss_fused": (k2, bytes_fused, T),
                "k3_ewma_update": (k3, bytes_k3, args.ewma_n)}
        alt = {"path": "two-call", "ms": round((alt_k1 + alt_k2) * 1e3, 4),
               "k1_ms": round(alt_k1 * 1e3, 4), "k2_ms": round(alt_k2 * 1e3, 4),
               "tokens_per_s": round(world * T / (alt_k1 + alt_k2), 1),
               "hbm_frac": round((bytes_k1 + bytes_k2) / (alt_k1 + alt_k2) / 1e9 / peak, 4)}
        loss_bytes = bytes_fused
    else:
        kern = {"k1_token_logprob": (k1, bytes_k1, T), "k2_decoupled_loss_fwd_bwd": (k2, bytes_k2, T),
                "k3_ewma_update": (k3, bytes_k3, args.ewma_n)}
        alt = {"path": "fused", "ms": round(alt_k2 * 1e3, 4),
               "tokens_per_s": round(world * T / alt_k2, 1),
               "hbm_frac": round(bytes_fused / alt_k2 / 1e9 / peak, 4)}
        loss_bytes = bytes_k1 + bytes_k2
    roof = {}
    for name, (sec, byts, units) in kern.items():
        achieved = byts / sec / 1e9
        roof[name] = {
            "bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
            "frac": round(achieved / peak, 4), "peak_kind": peak_kind,
            "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
            "traffic": traffic_bytes(traffic, name, T, n_valid, args.ewma_n),
            "algorithmic_bytes": byts, "ms": round(sec * 1e3, 4),
        }
    dominant = max(roof, key=lambda k: roof[k]["ms"])
    loss_ms = (k1 + k2) * 1e3
    line = {
        "metric": METRIC,
        "value": round(world * T / (elapsed / args.steps), 1),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": dict(workload_config(args, batch, n_valid, world), loss_path=args.loss_path,
                       rho=round(st_last.rho, 5), ewma_resets_timed=resets),
        "roofline": dict(roof[dominant], kernel=dominant),
        "kernels": roof,
        "loss_only": {"path": args.loss_path, "tokens_per_s": round(world * T / (k1 + k2), 1),
                      "ms": round(loss_ms, 4),
                      "hbm_frac": round(loss_bytes / (k1 + k2) / 1e9 / peak, 4)},
        "loss_only_other_path": alt,
        "gpu_launches": args.steps * (5 if args.loss_path == "fused" else 6),
        "graph_replay": graph,
        "clocks": clk,
    }
    # e2e first: it pins 70 GB of host memory, which the oracle's float64
    # working set would otherwise have churned just before
    if not args.no_e2e:
        line["e2e"] = run_e2e(args, batch, theta, theta_prox, state, stats, loss, world, dev)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(batch, args.ewma_n, args.cpu_seconds)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def _anon_huge_bytes():
    """Anonymous memory of this host backed by transparent huge pages."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("AnonHugePages:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def _host_available_bytes():
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def run_e2e(args, batch, theta, theta_prox, state, stats, loss_fn, world, dev):
    """Same step through the public API with the inputs in pinned HOST memory:
    every step copies the logits, token arrays and the new actor parameters to
    the device and reads the loss statistics back.  The host link, not HBM,
    bounds this number; ``pipeline.HostFedStep`` runs the copies on their own
    stream with the kernels underneath."""
    import torch

    from paper_2605_12070_gb300 import dp, occ
    from paper_2605_12070_gb300.pipeline import HostFedStep
    loss_inputs = [batch.z_old, batch.z_theta, batch.ids, batch.logp_mu, batch.adv]
    if batch.mask is not None:
        loss_inputs.append(batch.mask)
    need = sum(t.numel() * t.element_size() for t in loss_inputs + [theta])
    # every rank on this host pins its own copy: check for all of them at once,
    # after a barrier so that no rank has allocated yet, and decide together
    local = int(os.environ.get("LOCAL_WORLD_SIZE", str(world)))
    if world > 1:
        torch.distributed.barrier()
    avail = _host_available_bytes()
    fits = torch.tensor([1 if avail >= 1.3 * need * local else 0], device=dev)
    if world > 1:
        torch.distributed.all_reduce(fits, op=torch.distributed.ReduceOp.MIN)
    if not int(fits.item()):
        return {"value": None, "unit": "tokens/s",
                "skipped": f"needs {local} x {need / 1e9:.0f} GB of pinned host memory, "
                           f"{avail / 1e9:.0f} GB available"}
    # page-locked, huge-page backed: the host link's address translation over
    # 70 GB of buffers is the difference between ~100 and ~165 GB/s on some hosts
    huge0 = _anon_huge_bytes()
    host = [occ.occ_host_alloc(tuple(t.shape), t.dtype) for t in loss_inputs + [theta]]
    for h, d in zip(host, loss_inputs + [theta]):
        h.copy_(d)
    huge = _anon_huge_bytes() - huge0
    stats_h = torch.empty(occ.LOSS_STATS_BYTES, dtype=torch.uint8, pin_memory=True)
    stream = torch.cuda.current_stream(dev)

    def ewma():
        if world > 1:
            dp.allreduce_loss_stats(stats)
        occ.occ_ewma_update(theta_prox, theta, EWMA_BETA, state, stats=stats, tau=args.tau)

    pipe = HostFedStep(loss_inputs, theta, loss_fn, ewma,
                       after_step=lambda: stats_h.copy_(stats, non_blocking=True), stream=stream)
    pipe.step(host[:-1], host[-1])
    torch.cuda.synchronize()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(stream)
    pipe.start_timing(s)
    for _ in range(args.e2e_steps):
        pipe.step(host[:-1], host[-1])
    e.record(stream)
    torch.cuda.synchronize()
    sec = s.elapsed_time(e) / 1e3 / args.e2e_steps
    # the host link alone on this machine, right after: the same bytes copied
    # back to back from the same pinned buffers, no kernels
    s.record(stream)
    for _ in range(args.e2e_steps):
        for h, d in zip(host, loss_inputs + [theta]):
            d.copy_(h, non_blocking=True)
    e.record(stream)
    torch.cuda.synchronize()
    copy_sec = s.elapsed_time(e) / 1e3 / args.e2e_steps
    if world > 1:
        t = torch.tensor([sec, copy_sec], dtype=torch.float64, device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        sec, copy_sec = float(t[0].item()), float(t[1].item())
    occ.decode_loss_stats(stats_h)
    return {"value": round(world * batch.T / sec, 1), "unit": "tokens/s",
            "h2d_bytes_per_step": need, "d2h_bytes_per_step": occ.LOSS_STATS_BYTES,
            "ms_per_step": round(sec * 1e3, 3), "steps": args.e2e_steps,
            "h2d_gbs": round(need / sec / 1e9, 1),
            "h2d_copy_only_gbs": round(need / copy_sec / 1e9, 1),
            "host_buffers": "occ_host_alloc (huge pages)",
            "host_huge_page_fraction": round(min(1.0, max(0.0, huge / need)), 3),
            "overlap": "copies on a second stream; loss and EWMA kernels run under them"}


def run_ewma_variants(args, dev):
    """Times the bf16 proximal buffer (nearest and stochastic rounding, fp32 and
    bf16 theta) on --ewma-n parameters and the pinned-host buffer on 2e9."""
    import torch

    from paper_2605_12070_gb300 import occ
    from paper_2605_12070_gb300.workloads import make_ewma_buffers

    def timeit(fn, reps=5, warm=2):
        for _ in range(warm):
            fn()
        torch.cuda.synchronize()
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s.record()
        for _ in range(reps):
            fn()
        e.record()
        torch.cuda.synchronize()
        return s.elapsed_time(e) / reps

    peak, peak_kind = measured_peak()
    n = args.ewma_n
    th, tp = make_ewma_buffers(n, seed=0, device=dev)
    tpb = tp.to(torch.bfloat16)
    del tp
    st = occ.new_ewma_state(dev, w0=1.0 / (1.0 - EWMA_BETA))
    out = {"metric": "PPO-EWMA update variants", "unit": "ms", "n_params": n,
           "peak_gbs": peak, "peak_kind": peak_kind}
    for name, fn, bpp in (
            ("bf16_buffer_f32_theta_nearest",
             lambda: occ.occ_ewma_update_bf16(tpb, th, EWMA_BETA, st, sr_seed=0), 8),
            ("bf16_buffer_f32_theta_stochastic",
             lambda: occ.occ_ewma_update_bf16(tpb, th, EWMA_BETA, st, sr_seed=77), 8)):
        ms = timeit(fn)
        out[name] = {"ms": round(ms, 3), "frac": round(n * bpp / ms / 1e6 / peak, 4)}
    thb = th.to(torch.bfloat16)
    del th
    ms = timeit(lambda: occ.occ_ewma_update_bf16(tpb, thb, EWMA_BETA, st, sr_seed=77))
    out["bf16_buffer_bf16_theta_stochastic"] = {"ms": round(ms, 3),
                                                "frac": round(n * 6 / ms / 1e6 / peak, 4)}
    del tpb
    m = min(n, 2_000_000_000)
    host = occ.occ_host_alloc((m,), torch.bfloat16)
    host.copy_(thb[:m])
    staging = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    s1 = torch.cuda.Stream(dev)
    ms = timeit(lambda: occ.occ_ewma_update_host(host, thb[:m], EWMA_BETA, st, staging, sr_seed=5,
                                                 stream1=s1), reps=3, warm=1)
    out["host_bf16_buffer"] = {"ms": round(ms, 3), "n_params": m, "staging_bytes": 256 << 20,
                               "host_device_gbs": round(2 * m * 2 / ms / 1e6, 1)}
    print(json.dumps(out), flush=True)


def workload_config(args, batch, n_valid, world):
    """The workload part of the JSON line's config, shared by both arms."""
    T, V = batch.T, batch.V
    dt = str(batch.z_theta.dtype).replace("torch.", "")
    es = batch.z_theta.element_size()
    return {
        "workload": (f"decoupled-loss step on the {args.workload} batch, T={T} tokens "
                     f"({n_valid} valid), V={V} {dt} old and current logits (log pi_old, loss "
                     f"fwd + dlogits) chained with the PPO-EWMA update of {args.ewma_n} fp32 "
                     f"parameters"),
        "T": T, "V": V, "ewma_params": args.ewma_n, "logits_dtype": dt,
        "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
        "l2": (f"inputs larger than L2 ({2 * T * V * es / 1e9:.0f} GB logits, "
               f"{8 * args.ewma_n / 1e9:.0f} GB EWMA buffers): no flush"),
        "rd_band": [batch.rd_lo, batch.rd_hi], "eps": [batch.eps_low, batch.eps_high],
        "tau": args.tau,
    }


def run_reference(args, batch, world):
    """The oracle as the reference arm.  Each step is a real, bounded sample of
    the workload: the float64 oracle on REF_SAMPLE_TOKENS tokens of the batch
    and the matching share of the EWMA parameters, on the host cores; the
    line's ms_per_step is the time those steps took, and value is the tokens
    they processed per second."""
    import numpy as np

    rng = np.random.default_rng(1)
    S, P, _, threads = oracle_steps(batch, args.ewma_n, rng, steps=args.warmup)
    S, P, times, threads = oracle_steps(batch, args.ewma_n, rng, steps=args.steps)
    step_s = sum(times) / len(times)
    value = S / step_s
    n_valid = batch.T if batch.mask is None else int(batch.mask.sum().item())
    sample = (f"per step: float64 oracle on {S} tokens drawn from the T={batch.T}, V={batch.V} "
              f"batch (log pi_old, loss, dlogits) and {P} EWMA parameters (the step's "
              f"parameters-per-token), {threads} threads")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(step_s * 1e3, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": dict(workload_config(args, batch, n_valid, world), loss_path="oracle",
                       sample_tokens_per_step=S, sample_ewma_params_per_step=P),
        "full_step_s_extrapolated": round(batch.T / value, 2),
        "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": threads,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "repo_libs_loaded": repo_libs_loaded(),
    }
    print(json.dumps(line), flush=True)


def repo_libs_loaded():
    """Shared objects of this repository mapped into the process (from
    /proc/self/maps; empty where that file does not exist)."""
    found = set()
    try:
        with open("/proc/self/maps") as f:
            for line in f:
                path = line.split()[-1] if len(line.split()) >= 6 else ""
                if path.startswith(ROOT) and ".so" in os.path.basename(path):
                    found.add(os.path.relpath(path, ROOT))
    except OSError:
        pass
    return sorted(found)


if __name__ == "__main__":
    main()
