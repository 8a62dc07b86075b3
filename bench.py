"""Benchmark: one FastRL kept-token GRPO step per iteration on GB300.

A step is the whole data-parallel path on one batch: grpo_advantage -> grpo_prune ->
grpo_compact -> (host: kept counts, adaptive rollout count) -> grpo_loss_fwd_bwd over the kept
tokens.  The default workload is the Qwen2.5-vocabulary batch: 16 prompts x G=8 rollouts,
lognormal completion lengths (median 384, capped at 1024), V = 152064, bf16 logits with a
Zipf(1.1) rank bias plus N(0, 2^2) noise, keep ratio 0.5, bf16 dlogits.  The logits of every
token (~16 GB) are resident before timing; the loss reads only the kept rows.

Output: one JSON line (rank 0).  `value` is kept tokens per second over all ranks (device
time, CUDA events); `e2e` repeats the step from inputs in pinned host memory (the selection
inputs copied whole, then only the kept rollouts' logit rows) with the loss read back, all inside
the timed region; `roofline` relates the loss kernel's event-timed
duration to the measured HBM copy bandwidth; `cpu_baseline` times the fp64 oracle on a bounded
sample on this machine's host cores.  `--impl reference` times that oracle as the reference
arm.  Under torchrun each rank runs its own batch (weak scaling); the only collectives are the
barrier and the max-over-ranks timing.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "kept-token GRPO loss fwd+bwd tokens/s and logits HBM GB/s (% of GB300 peak)"
UNIT = "kept tokens/s"
SIDE_BYTES_PER_ROW = 36  # y, old, ref, logp (4 each), src_token 8, row rollout 4, row loss 8
# GSPO: forward (src 8, y 4, logp 4, stats 16), sequence pass (src 8, logp, old, ref, coef 4
# each), dlogits pass (src 8, coef 4, stats 16, y 4)
GSPO_SIDE_BYTES_PER_ROW = 88
FALLBACK_HBM_GBS = 6800.0
# rough step times of the further workloads (ms), to size their timed step counts
EXTRA_MS_GUESS = {"large": 5.2, "long": 20.0, "small": 0.26, "tiny": 0.07}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="qwen", help="tiny|small|qwen|large|long or 0-4")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--prompts", type=int, default=0,
                    help="override the workload's prompt count (a smaller case for profiling)")
    ap.add_argument("--group", type=int, default=0,
                    help="override the rollouts per prompt G (a smaller case for profiling)")
    ap.add_argument("--loss", choices=["grpo", "gspo", "lmhead", "lmhead-gspo"], default="grpo",
                    help="grpo: Eq. 1's token-level ratio (fused, one pass); gspo: the sequence-level "
                         "ratio of FastRL's GSPO variant (three passes, host-synced); lmhead: the "
                         "output layer fused with the token loss (hidden states in, logits on the "
                         "tensor cores, dhidden and dweight out); lmhead-gspo: the same with GSPO's "
                         "sequence-level loss (clip 3e-4 / 4e-4, beta 0)")
    ap.add_argument("--hidden", type=int, default=0,
                    help="hidden size of the output layer with --loss lmhead (default 3584)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-lmhead", action="store_true",
                    help="skip the default run's side measurement of the output layer fused with "
                         "the loss (tensor cores)")
    ap.add_argument("--no-graph", action="store_true",
                    help="run each step's calls directly instead of replaying captured CUDA graphs")
    ap.add_argument("--extra-configs", default="large,long",
                    help="with the qwen workload: further workloads measured after it, each in "
                         "its own sub-record of the line (comma-separated; empty for none)")
    ap.add_argument("--extra-seconds", type=float, default=0.5,
                    help="timed device seconds per further workload (sets its step count)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def workload_desc(w, T, T_kept, K):
    return {
        "workload": "%s: %d prompts x G=%d rollouts, lengths %s, V=%d, %s logits (%s), rewards %s,"
                    " %.0f%% zero-advantage groups, keep ratio %.2f (cap %d/prompt), %s dlogits"
                    % (w.name, w.P, w.G, w.length, w.V, w.logits_dtype, w.logits_kind,
                       w.reward_kind, 100 * w.zero_adv_frac, w.keep_ratio, w.keep_cap,
                       w.dlogits_dtype),
        "V": w.V, "prompts": w.P, "G": w.G, "T_tokens": T, "T_kept": T_kept, "kept_rollouts": K,
        "eps": w.eps, "beta": w.beta, "tau": w.tau, "ngram_n": w.ngram_n,
        "io": "%s logits -> %s dlogits" % (w.logits_dtype, w.dlogits_dtype),
        "l2": "inputs larger than L2 (logits %.1f GB vs 129 MB L2); no flush" % (T * w.V * w.in_bytes / 1e9),
    }


def measured_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs, copy read+write)"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback 6.8 TB/s (no MEASURED_PEAKS.json)"


def code_hash(files, root=None):
    """Hash of the code of `files` (under paper_2609_36932_gb300/csrc): comments, blank lines and
    the host-side NVTX markers (GRPO_TRACE and its header) removed, so that an edit which leaves
    the kernels alone does not orphan a profile taken on them."""
    import re
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(root or ROOT, "paper_2609_36932_gb300", "csrc", f)) as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        lines = [ln.rstrip() for ln in text.splitlines()
                 if ln.strip() and "GRPO_TRACE" not in ln and '"trace.cuh"' not in ln]
        h.update("\n".join(lines).encode())
    return h.hexdigest()[:16]


def loss_source_hash(root=None):
    return code_hash(("loss.cu", "gspo.cu", "rowops.cuh", "common.cuh"), root)


def profiled_traffic(workload_name, rows, launches=1):
    """DRAM bytes of a loss call over `rows` kept rows in `launches` kernel launches, from the
    committed ncu record of the current kernel source (else None): bytes per kept row times the
    rows, less the per-launch residue (dlogits lines still dirty in L2 when a launch ends) where
    the record has one, fitted from captures of two sizes."""
    p = os.path.join(ROOT, "profiles", "loss_kernel_traffic.json")
    try:
        with open(p) as f:
            d = json.load(f)
    except Exception:
        return None
    e = d.get(workload_name)
    if not e or e.get("source_hash") != loss_source_hash():
        return None
    return float(e["dram_bytes_per_row"]) * rows - float(e.get("dram_bytes_residue", 0.0)) * launches


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + ",".join(self.FIELDS), "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.15)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
                pw.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[3:]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def host_mem_available():
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return float("inf")


def combine_ranks(elapsed_ms, kept, world, device):
    """(max over ranks of the timed region, sum over ranks of the kept tokens processed)."""
    if world <= 1:
        return float(elapsed_ms), float(kept)
    import torch
    import torch.distributed as dist
    mx = torch.tensor([float(elapsed_ms)], dtype=torch.float64, device=device)
    sm = torch.tensor([float(kept)], dtype=torch.float64, device=device)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx.item()), float(sm.item())


def rank_seed(base_seed, rank):
    """Each rank draws its own batch (weak scaling: per-rank work is fixed as ranks grow)."""
    return base_seed + rank


def build_inputs(w, seed, device):
    """Seeded synthetic batch, resident on `device` (logits of every token)."""
    import torch
    from paper_2609_36932_gb300 import workloads
    b = workloads.make_batch(w, seed)
    T = b["T"]
    rewards = torch.from_numpy(b["rewards"]).to(device)
    ids = torch.from_numpy(b["ids"]).to(device)
    off = torch.from_numpy(b["off"]).to(device)
    logits = workloads.logits_rows(w, seed, range(T), device)
    old, ref = workloads.old_ref_logp(logits, b["ids"], b["noise_old"], b["noise_ref"])
    return b, dict(rewards=rewards, ids=ids, off=off, logits=logits, old=old, ref=ref)


def make_step(w, dev_inputs, loss="grpo"):
    from paper_2609_36932_gb300.pipeline import GrpoStep, StepParams
    p = StepParams(G=w.G, V=w.V, ngram_n=w.ngram_n, tau=w.tau, keep_cap=w.keep_cap,
                   eps_low=w.eps, eps_high=w.eps, beta=w.beta, dlogits_dtype=w.dlogits_dtype,
                   chunk_rows=0 if loss == "gspo" else w.chunk_rows,
                   ratio_level="sequence" if loss == "gspo" else "token")
    d = dev_inputs
    return GrpoStep(p, d["rewards"], d["ids"], d["off"], d["logits"], d["old"], d["ref"])


def oracle_sample(w, b, rows_src, rows_rollout, T_kept, logits_rows_host, old, ref, threads=0):
    """Time the oracle: selection on the whole batch, then the loss on the given kept rows."""
    import oracle
    oracle.set_threads(threads)
    t0 = time.perf_counter()
    adv, _ = oracle.advantage(b["rewards"], w.G)
    keep, kpp = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
    comp = oracle.compact(keep, b["off"])
    t_sel = time.perf_counter() - t0
    n = len(rows_src)
    t1 = time.perf_counter()
    oracle.loss(logits_rows_host, w.V, b["ids"][rows_src], old[rows_src], ref[rows_src], adv,
                rows_rollout, eps_low=w.eps, eps_high=w.eps, beta=w.beta, denom_tokens=T_kept,
                dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0, n_rows=n)
    t_loss = time.perf_counter() - t1
    return t_sel, t_loss, comp, int(oracle.set_threads(0))


def host_logits_bits(t):
    import torch
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.float().cpu().numpy()


def cpu_baseline_ours(w, b, step, dev_inputs, target_s):
    """Oracle timed on a bounded sample of this workload (the first kept rows)."""
    src, rr = step.kept_rows()
    old = dev_inputs["old"].cpu().numpy()
    ref = dev_inputs["ref"].cpu().numpy()
    # calibrate on 8 rows, then size the sample for ~target_s seconds of loss work
    n0 = min(8, len(src))
    _, tl0, _, cores = oracle_sample(w, b, src[:n0], rr[:n0], step.T_kept,
                                     host_logits_bits(dev_inputs["logits"][src[:n0]]), old, ref)
    per_row = max(tl0 / max(n0, 1), 1e-6)
    n = int(min(len(src), max(n0, target_s / per_row)))
    rows = src[:n]
    t_sel, t_loss, _, cores = oracle_sample(w, b, rows, rr[:n], step.T_kept,
                                            host_logits_bits(dev_inputs["logits"][rows]), old, ref)
    t_per_token = t_loss / n + t_sel / max(step.T_kept, 1)
    out = {"value": 1.0 / t_per_token, "unit": UNIT, "cores": cores, "kind": "oracle",
           "sample": "fp64 oracle: advantage+prune+compact on the whole batch (%.2f s, amortised"
                     " over its %d kept tokens) + loss fwd/bwd on the first %d kept rows (%.2f s)"
                     % (t_sel, step.T_kept, n, t_loss)}
    # the same oracle on one core, on the first rows of the same sample (about target_s / 2)
    n1 = int(min(n, max(n0, 0.5 * target_s / (per_row * max(cores, 1)))))
    rows1 = src[:n1]
    import oracle
    try:
        oracle.set_threads(1)
        t_sel1, t_loss1, _, c1 = oracle_sample(w, b, rows1, rr[:n1], step.T_kept,
                                               host_logits_bits(dev_inputs["logits"][rows1]),
                                               old, ref)
    finally:
        oracle.set_threads(cores)
    out["single_thread"] = {
        "value": 1.0 / (t_loss1 / n1 + t_sel1 / max(step.T_kept, 1)), "unit": UNIT, "cores": c1,
        "sample": "the same oracle with one OpenMP thread: selection on the whole batch (%.2f s)"
                  " + loss fwd/bwd on the first %d kept rows (%.2f s)" % (t_sel1, n1, t_loss1)}
    return out


def cpu_baseline_gspo(w, b, step, dev_inputs, target_s):
    """GSPO's oracle timed on a bounded sample: selection on the whole batch, then the sequence-
    level loss over the first kept sequences (whole sequences: a ratio needs all of its rows)."""
    import torch
    import oracle
    cores = int(oracle.set_threads(0))
    t0 = time.perf_counter()
    adv, _ = oracle.advantage(b["rewards"], w.G)
    keep, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
    comp = oracle.compact(keep, b["off"])
    t_sel = time.perf_counter() - t0
    K, T_kept = comp["K"], comp["T_kept"]
    if K == 0 or T_kept == 0:
        return None
    kept_idx, kept_off = comp["kept_idx"][:K], comp["kept_off"][:K + 1]
    old = dev_inputs["old"].cpu().numpy()
    ref = dev_inputs["ref"].cpu().numpy()
    dev = dev_inputs["logits"].device

    def run(nseq):
        rows = comp["src_token"][:kept_off[nseq]]
        bits = host_logits_bits(dev_inputs["logits"][torch.from_numpy(rows).to(dev)])
        t = time.perf_counter()
        oracle.gspo_loss(bits, w.V, b["ids"][rows], old[rows], ref[rows], adv, kept_idx[:nseq],
                         kept_off[:nseq + 1], n_seq=K, eps_low=w.eps, eps_high=w.eps, beta=w.beta,
                         dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
        return time.perf_counter() - t, int(kept_off[nseq])

    k = 1
    while k < K and kept_off[k] == 0:
        k += 1
    t1, r1 = run(k)
    per_row = max(t1 / max(r1, 1), 1e-6)
    target_rows = target_s / per_row
    while k < K and kept_off[k + 1] <= target_rows:
        k += 1
    t, rows = run(k)
    t_per_token = t / max(rows, 1) + t_sel / max(T_kept, 1)
    return {"value": 1.0 / t_per_token, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "fp64 oracle: advantage+prune+compact on the whole batch (%.2f s, amortised"
                      " over its %d kept tokens) + GSPO's sequence-level loss on the first %d kept"
                      " sequences (%d rows, %.2f s)" % (t_sel, T_kept, k, rows, t)}


def run_reference_gspo(args, w, b, comp):
    """The reference arm for GSPO's loss: selection on the whole batch, then the sequence-level
    loss over the first whole kept sequences that fit the per-step time budget."""
    from paper_2609_36932_gb300 import workloads
    import oracle
    K, T_kept = comp["K"], comp["T_kept"]
    kept_idx, kept_off = comp["kept_idx"][:K], comp["kept_off"][:K + 1]

    def sample(k):
        rows = comp["src_token"][:kept_off[k]]
        lg = workloads.logits_rows(w, args.seed, rows, "cpu")
        o, r = workloads.old_ref_logp(lg, b["ids"][rows], b["noise_old"][rows], b["noise_ref"][rows])
        return rows, host_logits_bits(lg), o.numpy(), r.numpy()

    def run(k, data):
        rows, bits, o, r = data
        t0 = time.perf_counter()
        adv, _ = oracle.advantage(b["rewards"], w.G)
        kp, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
        oracle.compact(kp, b["off"])
        t1 = time.perf_counter()
        oracle.gspo_loss(bits, w.V, b["ids"][rows], o, r, adv, kept_idx[:k], kept_off[:k + 1],
                         n_seq=K, eps_low=w.eps, eps_high=w.eps, beta=w.beta,
                         dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
        return t1 - t0, time.perf_counter() - t1

    k = 1
    while k < K and kept_off[k] == 0:
        k += 1
    t_sel, t_loss = run(k, sample(k))
    budget = 120.0 / max(args.steps + args.warmup, 1)
    per_row = t_loss / max(int(kept_off[k]), 1)
    while k < K and (int(kept_off[k + 1]) * per_row + t_sel) <= budget:
        k += 1
    data = sample(k)
    rows = int(kept_off[k])
    cores = int(oracle.set_threads(0))
    times = []
    for i in range(args.warmup + args.steps):
        t_sel, t_loss = run(k, data)
        if i >= args.warmup:
            times.append(t_loss / rows + t_sel / T_kept)
    value = 1.0 / statistics.mean(times)
    cfg = dict(workload_desc(w, b["T"], T_kept, K), loss="gspo")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": None,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": cfg,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": "per step: fp64 oracle advantage+prune+compact on the whole batch"
                                   " (amortised over %d kept tokens) + GSPO's sequence-level loss on"
                                   " the first %d kept sequences (%d rows)" % (T_kept, k, rows)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def run_reference(args, w):
    """The reference arm: the fp64 oracle as it stands, on this machine's host cores."""
    import torch
    from paper_2609_36932_gb300 import workloads
    import oracle
    rank, world, _ = dist_env()
    if rank != 0:
        return
    b = workloads.make_batch(w, args.seed)
    keep, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
    comp = oracle.compact(keep, b["off"])
    T_kept = comp["T_kept"]
    src_all, rr_all = comp["src_token"], comp["token_rollout"]
    if args.loss == "gspo":
        return run_reference_gspo(args, w, b, comp)
    # a bounded sample of kept rows, generated on the host
    n = min(len(src_all), 4)
    lg = workloads.logits_rows(w, args.seed, src_all[:n], "cpu")
    old, ref = workloads.old_ref_logp(lg, b["ids"][src_all[:n]], b["noise_old"][src_all[:n]],
                                      b["noise_ref"][src_all[:n]])
    old_full = np.zeros(b["T"], np.float32)
    ref_full = np.zeros(b["T"], np.float32)
    old_full[src_all[:n]] = old.numpy()
    ref_full[src_all[:n]] = ref.numpy()
    bits = host_logits_bits(lg)
    t_sel, t_loss, _, cores = oracle_sample(w, b, src_all[:n], rr_all[:n], T_kept, bits, old_full, ref_full)
    # size each step's sample so the whole run stays within ~2 minutes
    budget = 120.0 / max(args.steps + args.warmup, 1)
    per_row = t_loss / n
    rows = int(max(1, min(len(src_all), (budget - t_sel) / per_row))) if budget > t_sel else 1
    rows = min(rows, 512)
    sel = src_all[:rows]
    lg = workloads.logits_rows(w, args.seed, sel, "cpu")
    o, r = workloads.old_ref_logp(lg, b["ids"][sel], b["noise_old"][sel], b["noise_ref"][sel])
    old_full[sel] = o.numpy()
    ref_full[sel] = r.numpy()
    bits = host_logits_bits(lg)
    times = []
    for i in range(args.warmup + args.steps):
        t_sel, t_loss, _, cores = oracle_sample(w, b, sel, rr_all[:rows], T_kept, bits, old_full, ref_full)
        if i >= args.warmup:
            times.append(t_loss / rows + t_sel / T_kept)
    value = 1.0 / statistics.mean(times)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": None,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": dict(workload_desc(w, b["T"], T_kept, comp["K"]),
                                            loss=args.loss),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": "per step: fp64 oracle advantage+prune+compact on the whole batch"
                                   " (amortised over %d kept tokens) + loss fwd/bwd on the first %d"
                                   " kept rows" % (T_kept, rows)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


LMHEAD_METRIC = ("kept-token GRPO step with the output layer fused: tokens/s and tensor-core "
                 "TFLOP/s (% of GB300 bf16 peak)")


def measured_tensor_peak(sustained):
    key = "bf16_tflops_sustained" if sustained else "bf16_tflops"
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)[key]), "measured (MEASURED_PEAKS.json %s, cuBLAS bf16)" % key
    except Exception:
        return (1700.0, "fallback 1.7 PFLOP/s sustained") if sustained else (
            1900.0, "fallback 1.9 PFLOP/s burst")


def lmhead_inputs(w, D, seed, device):
    import torch
    from paper_2609_36932_gb300 import workloads
    b = workloads.make_batch(w, seed)
    hid = workloads.lmhead_hidden(b["T"], D, seed, device)
    wt = workloads.lmhead_weight(w.V, D, seed, device)
    old, ref = workloads.lmhead_old_ref(hid, wt, b["ids"], b["noise_old"], b["noise_ref"])
    d = dict(rewards=torch.from_numpy(b["rewards"]).to(device),
             ids=torch.from_numpy(b["ids"]).to(device), off=torch.from_numpy(b["off"]).to(device),
             hidden=hid, weight=wt, old=old, ref=ref)
    return b, d


GSPO_LMHEAD = dict(eps_low=3e-4, eps_high=4e-4, beta=0.0)  # GSPO's published clip widths


def lmhead_desc(w, D, T, T_kept, K, gspo=False):
    cfg = workload_desc(w, T, T_kept, K)
    cfg["workload"] = ("%s with the output layer: %d prompts x G=%d rollouts, lengths %s, hidden "
                       "size D=%d, V=%d, bf16 hidden states N(0,1) and weight N(0,4/D), rewards %s,"
                       " %.0f%% zero-advantage groups, keep ratio %.2f (cap %d/prompt); bf16 "
                       "dhidden, f32 dweight" % (w.name, w.P, w.G, w.length, D, w.V, w.reward_kind,
                                                  100 * w.zero_adv_frac, w.keep_ratio, w.keep_cap))
    cfg["D"] = D
    cfg["io"] = "bf16 hidden [T_kept, D] and weight [V, D] -> bf16 dhidden, f32 dweight"
    cfg["l2"] = ("inputs larger than L2 (weight %.2f GB, dweight %.2f GB vs 129 MB L2); no flush"
                 % (w.V * D * 2 / 1e9, w.V * D * 4 / 1e9))
    cfg["loss"] = "lmhead-gspo" if gspo else "lmhead"
    if gspo:
        cfg.update(eps_low=GSPO_LMHEAD["eps_low"], eps_high=GSPO_LMHEAD["eps_high"], beta=0.0,
                   ratio="sequence (GSPO): the kept rollouts are the sequences")
    return cfg


def oracle_lmhead_sample(w, b, d, src, rr, T_kept, n, threads=0):
    """Time the oracle: selection on the whole batch, then the output layer + loss (logits,
    dhidden and dweight) on the first n kept rows."""
    import oracle
    oracle.set_threads(threads)
    import torch
    rows = torch.from_numpy(np.ascontiguousarray(src[:n])).to(d["hidden"].device)
    h = d["hidden"][rows].float().cpu().numpy()
    wt = d["weight"].double().cpu().numpy()
    old = d["old"].cpu().numpy()[src[:n]]
    ref = d["ref"].cpu().numpy()[src[:n]]
    t0 = time.perf_counter()
    adv, _ = oracle.advantage(b["rewards"], w.G)
    keep, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
    oracle.compact(keep, b["off"])
    t_sel = time.perf_counter() - t0
    t1 = time.perf_counter()
    oracle.lmhead_loss(h, wt, b["ids"][src[:n]], old, ref, adv, rr[:n], eps_low=w.eps,
                       eps_high=w.eps, beta=w.beta, denom_tokens=T_kept)
    return t_sel, time.perf_counter() - t1, int(oracle.set_threads(0))


def cpu_baseline_lmhead_gspo(w, b, d, step, target_s):
    """The oracle on a bounded sample: selection on the whole batch, then the output layer and
    GSPO's loss over the first whole kept sequences."""
    import torch
    import oracle
    cores = int(oracle.set_threads(0))
    t0 = time.perf_counter()
    adv, _ = oracle.advantage(b["rewards"], w.G)
    keep, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
    comp = oracle.compact(keep, b["off"])
    t_sel = time.perf_counter() - t0
    K, T_kept = comp["K"], comp["T_kept"]
    kept_idx, kept_off, src = comp["kept_idx"][:K], comp["kept_off"][:K + 1], comp["src_token"]
    w64 = d["weight"].double().cpu().numpy()
    old, ref = d["old"].cpu().numpy(), d["ref"].cpu().numpy()

    def run(k):
        rows = src[:int(kept_off[k])]
        h = d["hidden"][torch.from_numpy(rows).to(d["hidden"].device)].double().cpu().numpy()
        t = time.perf_counter()
        oracle.lmhead_gspo_loss(h, w64, b["ids"][rows], old[rows], ref[rows], adv, kept_idx[:k],
                                kept_off[:k + 1], n_seq=K, **GSPO_LMHEAD)
        return time.perf_counter() - t, len(rows)

    k = 1
    t1, r1 = run(k)
    per_row = max(t1 / max(r1, 1), 1e-6)
    while k < K and kept_off[k + 1] * per_row <= target_s:
        k += 1
    t, rows = run(k)
    return {"value": 1.0 / (t / max(rows, 1) + t_sel / max(T_kept, 1)), "unit": UNIT,
            "cores": cores, "kind": "oracle",
            "sample": "fp64 oracle: advantage+prune+compact on the whole batch (%.2f s, amortised"
                      " over its %d kept tokens) + output layer and GSPO's loss on the first %d"
                      " kept sequences (%d rows, %.2f s)" % (t_sel, T_kept, k, rows, t)}


def lmhead_side(w, b, step, seed, dev, reps=3):
    """The output layer fused with the loss on this batch's kept rows (hidden states of width
    LMHEAD_D drawn for the same tokens): one host-timed call block, reported beside the main
    line.  Returns a dict, or None when the output layer's inputs do not fit in device memory."""
    import torch
    import paper_2609_36932_gb300 as g
    from paper_2609_36932_gb300 import workloads
    D = workloads.LMHEAD_D
    need = (b["T"] * D * 2 + w.V * D * 6 + 14 * (1 << 30))
    free, _ = torch.cuda.mem_get_info(dev)
    if need > 0.8 * free:
        return None
    hid = workloads.lmhead_hidden(b["T"], D, seed, dev)
    wt = workloads.lmhead_weight(w.V, D, seed, dev)
    old, ref = workloads.lmhead_old_ref(hid, wt, b["ids"], b["noise_old"], b["noise_ref"])
    T_kept = step.T_kept
    rows = step.src_token[:T_kept]
    ids = torch.from_numpy(b["ids"]).to(dev)
    kw = dict(row_index=rows, n_rows=T_kept, eps_low=w.eps, eps_high=w.eps, beta=w.beta,
              denom_tokens=max(T_kept, 1))
    out = g.grpo_lmhead_loss_fwd_bwd(hid, wt, ids, old, ref, step.adv, step.token_rollout, **kw)
    ws, dh, dw = out["ws"], out["dhidden"], out["dweight"]
    g.grpo_lmhead_loss_fwd_bwd(hid, wt, ids, old, ref, step.adv, step.token_rollout, dhidden=dh,
                               dweight=dw, ws=ws, **kw)
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        g.grpo_lmhead_loss_fwd_bwd(hid, wt, ids, old, ref, step.adv, step.token_rollout,
                                   dhidden=dh, dweight=dw, ws=ws, **kw)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    # the same calls with the logits recomputed in a second tensor-core pass (the other setting)
    g.grpo_lmhead_tune(0, 0, 1)
    try:
        g.grpo_lmhead_loss_fwd_bwd(hid, wt, ids, old, ref, step.adv, step.token_rollout,
                                   dhidden=dh, dweight=dw, ws=ws, **kw)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            g.grpo_lmhead_loss_fwd_bwd(hid, wt, ids, old, ref, step.adv, step.token_rollout,
                                       dhidden=dh, dweight=dw, ws=ws, **kw)
        e1.record(stream)
        torch.cuda.synchronize()
    finally:
        g.grpo_lmhead_tune(0, 0, 0)
    ms_rec = e0.elapsed_time(e1) / reps
    peak, src = measured_tensor_peak(sustained=True)
    tf = 6.0 * T_kept * w.V * D / (ms / 1e3) / 1e12
    del hid, wt, old, ref, dh, dw, ws, out
    torch.cuda.empty_cache()
    return {"call": "grpo_lmhead_loss_fwd_bwd", "D": D, "T_kept": T_kept, "calls": reps,
            "ms_per_call": ms, "kept_tokens_per_s": T_kept / (ms / 1e3), "achieved": tf,
            "unit": "TFLOP/s", "peak": peak, "frac": tf / peak, "peak_source": src,
            "ms_per_call_recomputed_logits": ms_rec,
            "note": "the output layer fused with the loss on this batch's kept rows: logits "
                    "h W^T on the tcgen05 tensor cores (f32 logits kept one chunk at a time), "
                    "loss, dlogits, dhidden, dweight; 6 T_kept V D algorithmic FLOPs per call "
                    "(forward logits and the two products); ms_per_call_recomputed_logits: the "
                    "same call recomputing the logits in a second tensor-core pass instead "
                    "(grpo_lmhead_tune); bench.py --loss lmhead runs it as a step"}


def lmhead_products(d, step, T_kept, V, D, peak, peak_src, nrep=3):
    """The two backward products alone (grpo_lmhead_grad) on the step's kept rows: dlogits taken
    from one fused call, the kept hidden rows gathered densely; each product event-timed on this
    stream against the burst tensor peak (2 T V D FLOPs each)."""
    import torch
    import paper_2609_36932_gb300 as g
    free, _ = torch.cuda.mem_get_info(d["hidden"].device)
    ldd = g.grpo_lmhead_dlogits_stride(V)
    if T_kept == 0 or T_kept * ldd * 2 + V * D * 4 + 2 * T_kept * D * 4 > 0.8 * free:
        return None
    dl = torch.empty((T_kept, ldd), dtype=torch.bfloat16, device=d["hidden"].device)
    p = step.p
    g.grpo_lmhead_loss_fwd_bwd(d["hidden"], d["weight"], d["ids"], d["old"], d["ref"], step.adv,
                               step.token_rollout, row_index=step.src_token[:T_kept],
                               n_rows=T_kept, eps_low=p.eps_low, eps_high=p.eps_high, beta=p.beta,
                               denom_tokens=T_kept, dlogits_out=dl)
    hk = d["hidden"][step.src_token[:T_kept]].contiguous()
    dlv = dl[:, :V]
    out = {}
    stream = torch.cuda.current_stream()
    for name, kw in (("dhidden", dict(want_dweight=False)), ("dweight", dict(want_dhidden=False))):
        r = g.grpo_lmhead_grad(dlv, hk, d["weight"], **kw)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(nrep):
            g.grpo_lmhead_grad(dlv, hk, d["weight"], dhidden=r["dhidden"], dweight=r["dweight"],
                               ws=r["ws"], **kw)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / nrep
        tf = 2.0 * T_kept * V * D / (ms / 1e3) / 1e12
        out[name] = {"ms": ms, "achieved": tf, "frac": tf / peak}
        del r
    del dl, hk
    torch.cuda.empty_cache()
    out.update({"unit": "TFLOP/s", "peak": peak, "peak_source": peak_src, "calls": nrep,
                "kernel": "gemm_bf16_kernel (tcgen05, gemm.cu) through grpo_lmhead_grad",
                "note": "dhidden = dlogits W and dweight = dlogits^T h over all kept rows in one "
                        "call each (the fused call runs them per dlogits chunk)"})
    return out


def run_lmhead(args, w):
    """--loss lmhead: the step with the output layer fused (GrpoStep in output-layer mode)."""
    import torch
    import torch.distributed as dist
    import paper_2609_36932_gb300 as g
    from paper_2609_36932_gb300 import workloads
    from paper_2609_36932_gb300.pipeline import GrpoStep, StepParams

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    g.lib()
    D = args.hidden or workloads.LMHEAD_D
    gspo = args.loss == "lmhead-gspo"
    b, d = lmhead_inputs(w, D, rank_seed(args.seed, rank), dev)
    if gspo:
        p = StepParams(G=w.G, V=w.V, ngram_n=w.ngram_n, tau=w.tau, keep_cap=w.keep_cap,
                       ratio_level="sequence", **GSPO_LMHEAD)
    else:
        p = StepParams(G=w.G, V=w.V, ngram_n=w.ngram_n, tau=w.tau, keep_cap=w.keep_cap,
                       eps_low=w.eps, eps_high=w.eps, beta=w.beta)
    step = GrpoStep(p, d["rewards"], d["ids"], d["off"], None, d["old"], d["ref"],
                    hidden=d["hidden"], weight=d["weight"])
    for _ in range(max(args.warmup, 3)):
        step.run()
    torch.cuda.synchronize()
    K = args.steps
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0 = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    l0 = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    l1 = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    if local == 0:
        sampler.start()
        time.sleep(0.3)
    launches0 = g.grpo_kernel_launches()
    kept = 0
    ev0.record(stream)
    for i in range(K):
        s0[i].record(stream)
        step.select()
        l0[i].record(stream)
        step.loss_step()
        l1[i].record(stream)
        kept += step.T_kept
    ev1.record(stream)
    torch.cuda.synchronize()
    launches = g.grpo_kernel_launches() - launches0
    clocks = sampler.stop() if local == 0 else None
    g.check_status(step.status)
    elapsed_ms = ev0.elapsed_time(ev1)
    loss_ms = statistics.mean(a.elapsed_time(z) for a, z in zip(l0, l1))
    select_ms = statistics.mean(a.elapsed_time(z) for a, z in zip(s0, l0))
    elapsed_ms, kept_all = combine_ranks(elapsed_ms, kept, world, dev)
    value = kept_all / (elapsed_ms / 1e3)
    T_kept = step.T_kept
    flops_pass = 2.0 * T_kept * w.V * D

    # roofline of the pass-1 tile kernel: the same kept rows through grpo_lmhead_logp_fwd (that
    # kernel plus a row kernel of T_kept threads), event-timed on this stream
    lp = torch.empty(max(T_kept, 1), dtype=torch.float32, device=dev)
    rows_src = step.src_token[:T_kept]
    fw = g.grpo_lmhead_logp_fwd(d["hidden"], d["weight"], d["ids"], row_index=rows_src,
                                n_rows=T_kept, logp_out=lp)
    for _ in range(2):
        g.grpo_lmhead_logp_fwd(d["hidden"], d["weight"], d["ids"], row_index=rows_src,
                               n_rows=T_kept, logp_out=lp, ws=fw["ws"])
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    nrep = 5
    torch.cuda.synchronize()
    f0.record(stream)
    for _ in range(nrep):
        g.grpo_lmhead_logp_fwd(d["hidden"], d["weight"], d["ids"], row_index=rows_src,
                               n_rows=T_kept, logp_out=lp, ws=fw["ws"])
    f1.record(stream)
    torch.cuda.synchronize()
    f_ms = f0.elapsed_time(f1) / nrep
    peak, peak_src = measured_tensor_peak(sustained=False)
    peak_s, peak_s_src = measured_tensor_peak(sustained=True)
    achieved = flops_pass / (f_ms / 1e3) / 1e12
    roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                # pass 1 reads the weight once per group of row-block pairs: its DRAM bytes do
                # not scale per row from a small capture, and full-size captures are not taken
                "frac": achieved / peak, "traffic": None,
                "kernel": "lmhead_tile_kernel<pass 1> (+ gather and row kernels), timed through "
                          "grpo_lmhead_logp_fwd on the step's kept rows",
                "algorithmic_flops_per_launch": flops_pass, "launch_ms": f_ms,
                "peak_source": peak_src}
    step_tc = {"flops_per_step": 3 * flops_pass, "loss_ms": loss_ms,
               "achieved": 3 * flops_pass / (loss_ms / 1e3) / 1e12, "unit": "TFLOP/s",
               "peak": peak_s, "frac": 3 * flops_pass / (loss_ms / 1e3) / 1e12 / peak_s,
               "peak_source": peak_s_src,
               "note": "the whole fused call against its algorithmic work: the forward logits "
                       "and the dhidden and dweight products (2 T V D each), all on the "
                       "library's tcgen05 kernels; "
                       + ("GSPO's entry keeps the first chunk's f32 logits and recomputes the "
                          "later chunks' in a second pass" if gspo else
                          "the token loss keeps each chunk's f32 logits from pass 1 and forms "
                          "dlogits from them in a streaming pass")}
    products = None if gspo else lmhead_products(d, step, T_kept, w.V, D, peak, peak_src)

    # end to end: selection inputs, log-probs and hidden states from pinned host memory (hidden
    # rows of the kept rollouts only), loss read back, inside the timed region
    e2e = None
    names = ["rewards", "ids", "off", "old", "ref", "hidden"]
    if args.e2e_steps > 0:
        host = {}
        for k in names:
            host[k] = torch.empty(d[k].shape, dtype=d[k].dtype, pin_memory=True)
            host[k].copy_(d[k])
        loss_host = torch.empty(1, dtype=torch.float64, pin_memory=True)
        step.run_from_host(host, loss_host)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        kept_e, h2d_e, d2h_e = 0, 0, 0
        e0.record(stream)
        for _ in range(args.e2e_steps):
            hb, db = step.run_from_host(host, loss_host)
            h2d_e += hb
            d2h_e += db
            kept_e += step.T_kept
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms, kept_e = combine_ranks(e0.elapsed_time(e1), kept_e, world, dev)
        e2e = {"value": kept_e / (e_ms / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d_e // args.e2e_steps),
               "d2h_bytes_per_step": int(d2h_e // args.e2e_steps), "steps": args.e2e_steps,
               "transfer": "selection inputs and per-token log-probs whole; hidden states of the "
                           "kept rollouts only (grpo_upload_kept), after the selection; the "
                           "output-layer weight is a resident model parameter"}
        del host

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and gspo:
        cpu = cpu_baseline_lmhead_gspo(w, b, d, step, args.cpu_seconds)
    elif rank == 0 and world == 1 and not args.no_cpu_baseline:
        src, rr = step.kept_rows()
        n0 = min(16, len(src))  # a full row per worker thread for the calibration
        _, tl0, _ = oracle_lmhead_sample(w, b, d, src, rr, T_kept, n0)
        n = int(min(len(src), max(n0, args.cpu_seconds / max(tl0 / n0, 1e-6))))
        t_sel, t_loss, cores = oracle_lmhead_sample(w, b, d, src, rr, T_kept, n)
        cpu = {"value": 1.0 / (t_loss / n + t_sel / max(T_kept, 1)), "unit": UNIT, "cores": cores,
               "kind": "oracle",
               "sample": "fp64 oracle: advantage+prune+compact on the whole batch (%.2f s, "
                         "amortised over its %d kept tokens) + output layer and loss (logits, "
                         "dhidden, dweight) on the first %d kept rows (%.2f s)"
                         % (t_sel, T_kept, n, t_loss)}

    if rank == 0:
        line = {
            "metric": LMHEAD_METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": elapsed_ms / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded; the qwen batch with random-init output layer)",
            "config": lmhead_desc(w, D, b["T"], T_kept, step.K, gspo),
            "gpu_launches": int(launches), "cuda_graph": False,
            "roofline": roofline, "step_tensor": step_tc, "backward_products": products,
            "e2e": e2e, "cpu_baseline": cpu,
            "clocks": clocks,
            "path_overhead": {"select_ms": select_ms, "other_ms": elapsed_ms / K - select_ms - loss_ms},
            "loss_value": float(step.loss.item()), "ars_next_rollouts": step.n_next,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def run_reference_lmhead(args, w):
    """The reference arm for --loss lmhead: the fp64 oracle on this machine's host cores; each
    step runs the selection on the whole batch and the output layer + loss on a bounded sample
    of kept rows (inputs generated on the host)."""
    import torch
    from paper_2609_36932_gb300 import workloads
    import oracle
    D = args.hidden or workloads.LMHEAD_D
    gspo = args.loss == "lmhead-gspo"
    b = workloads.make_batch(w, args.seed)
    keep, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
    comp = oracle.compact(keep, b["off"])
    T_kept = comp["T_kept"]
    src, rr = comp["src_token"], comp["token_rollout"]
    K = comp["K"]
    kept_idx, kept_off = comp["kept_idx"][:K], comp["kept_off"][:K + 1]
    wt = workloads.lmhead_weight(w.V, D, args.seed, "cpu")
    w64 = wt.double().numpy()

    def sample(n):
        h = workloads.lmhead_hidden(b["T"], D, args.seed, "cpu", rows=src[:n])
        o, r = workloads.lmhead_old_ref(h, wt, b["ids"][src[:n]], b["noise_old"][src[:n]],
                                        b["noise_ref"][src[:n]])
        return h.float().numpy(), o.numpy(), r.numpy()

    def run(n, data):
        h, o, r = data
        t0 = time.perf_counter()
        adv, _ = oracle.advantage(b["rewards"], w.G)
        kp, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau, w.keep_cap, 1)
        oracle.compact(kp, b["off"])
        t1 = time.perf_counter()
        if gspo:  # n counts whole kept sequences
            oracle.lmhead_gspo_loss(h, w64, b["ids"][src[:kept_off[n]]], o, r, adv, kept_idx[:n],
                                    kept_off[:n + 1], n_seq=K, **GSPO_LMHEAD)
        else:
            oracle.lmhead_loss(h, w64, b["ids"][src[:n]], o, r, adv, rr[:n], eps_low=w.eps,
                               eps_high=w.eps, beta=w.beta, denom_tokens=T_kept)
        return t1 - t0, time.perf_counter() - t1

    rows_of = (lambda n: int(kept_off[n])) if gspo else (lambda n: n)
    first = 1
    while gspo and first < K and kept_off[first] == 0:
        first += 1
    t_sel, t_loss = run(first, sample(rows_of(first)))
    budget = 120.0 / max(args.steps + args.warmup, 1)
    if gspo:
        n = first
        per_row = t_loss / max(rows_of(first), 1)
        while n < K and rows_of(n + 1) <= 64 and rows_of(n + 1) * per_row + t_sel <= budget:
            n += 1
    else:
        n = int(max(1, min(len(src), 64, (budget - t_sel) / max(t_loss, 1e-6)))) if budget > t_sel else 1
    data = sample(rows_of(n))
    cores = int(oracle.set_threads(0))
    times = []
    for i in range(args.warmup + args.steps):
        t_sel, t_loss = run(n, data)
        if i >= args.warmup:
            times.append(t_loss / max(rows_of(n), 1) + t_sel / T_kept)
    value = 1.0 / statistics.mean(times)
    what = ("GSPO's loss on the first %d kept sequences (%d rows)" % (n, rows_of(n)) if gspo
            else "loss on the first %d kept rows" % n)
    print(json.dumps({
        "impl": "reference", "metric": LMHEAD_METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": None,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": lmhead_desc(w, D, b["T"], T_kept, comp["K"], gspo),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": "per step: fp64 oracle advantage+prune+compact on the whole batch"
                                   " (amortised over %d kept tokens) + output layer and %s"
                                   % (T_kept, what)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def timed_steps(args, w, seed, world, local, dev, steps, warmup):
    """Build a workload's batch on the device, warm up, then time `steps` whole steps with CUDA
    events on the launching stream (barrier and synchronisation on both sides, max over ranks).
    Returns the step, its inputs and the measurements, `roofline` for the loss call included."""
    import torch
    import torch.distributed as dist
    import paper_2609_36932_gb300 as g
    b, d = build_inputs(w, seed, dev)
    step = make_step(w, d, args.loss)
    for _ in range(max(warmup, 3)):
        step.run()
    torch.cuda.synchronize()
    l_before = g.grpo_kernel_launches()
    step.run()
    torch.cuda.synchronize()
    launches_per_step = g.grpo_kernel_launches() - l_before
    use_graph = not args.no_graph and step.p.chunk_rows == 0
    if use_graph:
        step.capture()
        for _ in range(max(warmup, 3)):
            step.run_graph()

    K = steps
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0 = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    l0 = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    l1 = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    if local == 0:
        sampler.start()
        time.sleep(0.3)
    launches0 = g.grpo_kernel_launches()
    kept = 0
    ev0.record(stream)
    for i in range(K):
        s0[i].record(stream)
        if use_graph:  # the step as two graph replays; the host reads the counts at its end
            step.replay_select()
            l0[i].record(stream)
            step.replay_loss()
            l1[i].record(stream)
            step.finish()
        else:
            step.select()
            l0[i].record(stream)
            step.loss_step()
            l1[i].record(stream)
        kept += step.T_kept
    ev1.record(stream)
    torch.cuda.synchronize()
    launches = launches_per_step * K if use_graph else g.grpo_kernel_launches() - launches0
    clocks = sampler.stop() if local == 0 else None
    g.check_status(step.status)
    elapsed_ms = ev0.elapsed_time(ev1)
    loss_ms = statistics.mean(a.elapsed_time(z) for a, z in zip(l0, l1))
    select_ms = statistics.mean(a.elapsed_time(z) for a, z in zip(s0, l0))
    elapsed_ms, kept_all = combine_ranks(elapsed_ms, kept, world, dev)
    value = kept_all / (elapsed_ms / 1e3)

    # roofline of the dominant kernel (the fused loss), from its event-timed launches
    if args.loss == "gspo":  # two reads and one write of every kept row (no row has zero gradient
        # in these workloads: beta > 0)
        bytes_per_row = w.V * (2 * w.in_bytes + w.out_bytes) + GSPO_SIDE_BYTES_PER_ROW
        traffic = profiled_traffic(w.name + "/gspo", step.T_kept)
        kernel = ("GSPO loss: logp_stream_kernel with row statistics, "
                  "gspo_seq_kernel, gspo_dlogits_kernel, fixed-order sum")
    else:
        bytes_per_row = w.V * (w.in_bytes + w.out_bytes) + SIDE_BYTES_PER_ROW
        n_launch = -(-step.T_kept // step.p.chunk_rows) if step.p.chunk_rows else 1
        traffic = profiled_traffic(w.name, step.T_kept, n_launch)
        kernel = "grpo_loss_kernel (+ the fixed-order loss sum, one 8-CTA cluster)"
        if step.p.chunk_rows:
            kernel += "; %d calls of at most %d kept rows" % (
                -(-step.T_kept // step.p.chunk_rows), step.p.chunk_rows)
    achieved = step.T_kept * bytes_per_row / (loss_ms / 1e3) / 1e9
    peak, peak_src = measured_peak()
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak,
                "traffic": traffic,
                "kernel": kernel,
                "algorithmic_bytes_per_launch": step.T_kept * bytes_per_row,
                "bytes_per_kept_row": bytes_per_row,
                "launch_ms": loss_ms, "peak_source": peak_src}
    return dict(b=b, d=d, step=step, K=K, elapsed_ms=elapsed_ms, value=value, loss_ms=loss_ms,
                select_ms=select_ms, launches=launches, use_graph=use_graph, clocks=clocks,
                roofline=roofline)


def sub_record(args, w, r, warmup):
    """A further workload's line inside the main one: the same measurements, without the
    end-to-end, CPU-baseline and side legs."""
    step = r["step"]
    return {"value": r["value"], "unit": UNIT, "steps": r["K"], "warmup": warmup,
            "ms_per_step": r["elapsed_ms"] / r["K"], "cuda_graph": r["use_graph"],
            "gpu_launches": int(r["launches"]), "roofline": r["roofline"], "clocks": r["clocks"],
            "config": dict(workload_desc(w, r["b"]["T"], step.T_kept, step.K), loss=args.loss),
            "path_overhead": {"select_ms": r["select_ms"],
                              "other_ms": r["elapsed_ms"] / r["K"] - r["select_ms"] - r["loss_ms"]},
            "loss_value": float(step.loss.item())}


def main():
    args = parse()
    import dataclasses
    from paper_2609_36932_gb300 import workloads
    w = workloads.get(args.config)
    if args.prompts > 0:
        w = dataclasses.replace(w, P=args.prompts)
    if args.group > 0:
        w = dataclasses.replace(w, G=args.group)
    if args.impl == "reference":
        if args.loss in ("lmhead", "lmhead-gspo"):
            if dist_env()[0] == 0:
                run_reference_lmhead(args, w)
            return
        run_reference(args, w)
        return
    if args.loss in ("lmhead", "lmhead-gspo"):
        run_lmhead(args, w)
        return
    import torch
    import torch.distributed as dist
    import paper_2609_36932_gb300 as g

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    g.lib()

    r = timed_steps(args, w, rank_seed(args.seed, rank), world, local, dev, args.steps,
                    args.warmup)
    b, d, step = r["b"], r["d"], r["step"]
    K, elapsed_ms, loss_ms, select_ms = r["K"], r["elapsed_ms"], r["loss_ms"], r["select_ms"]
    peak = r["roofline"]["peak"]
    stream = torch.cuda.current_stream()

    # the logp-only forward over the same kept rows (old/reference policy evaluation); one read
    logp_fwd = None
    if w.chunk_rows == 0:
        lp_out = torch.empty(max(step.T_kept, 1), dtype=torch.float32, device=dev)
        rows_src = step.src_token[:step.T_kept]
        for _ in range(3):
            g.grpo_logp_fwd(d["logits"], d["ids"], row_index=rows_src, n_rows=step.T_kept,
                            logp_out=lp_out)
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        nrep = 20
        f0.record(stream)
        for _ in range(nrep):
            g.grpo_logp_fwd(d["logits"], d["ids"], row_index=rows_src, n_rows=step.T_kept,
                            logp_out=lp_out)
        f1.record(stream)
        torch.cuda.synchronize()
        f_ms = f0.elapsed_time(f1) / nrep
        f_bytes = step.T_kept * (w.V * w.in_bytes + 16)
        logp_fwd = {"kernel": "logp_stream_kernel", "launch_ms": f_ms,
                    "achieved": f_bytes / (f_ms / 1e3) / 1e9, "unit": "GB/s",
                    "frac": f_bytes / (f_ms / 1e3) / 1e9 / peak,
                    "kept_tokens_per_s": step.T_kept / (f_ms / 1e3),
                    "algorithmic_bytes_per_launch": f_bytes}

    lmhead = None
    if not args.no_lmhead and args.loss == "grpo" and w.chunk_rows == 0:
        lmhead = lmhead_side(w, b, step, rank_seed(args.seed, rank), dev)

    # end to end: inputs copied from pinned host memory, loss read back, inside the timed region
    e2e = None
    names = ["rewards", "ids", "off", "logits", "old", "ref"]
    h2d = sum(d[k].numel() * d[k].element_size() for k in names)
    # every rank of this host pins its own copy: the budget is shared, and all ranks must agree
    # (the end-to-end leg has a barrier and cross-rank reductions)
    local_ranks = max(1, int(os.environ.get("LOCAL_WORLD_SIZE", "1")))
    fits = h2d <= 0.6 * host_mem_available() / local_ranks
    if world > 1:
        flag = torch.tensor([1 if fits else 0], dtype=torch.int32, device=dev)
        dist.all_reduce(flag, op=dist.ReduceOp.MIN)
        fits = bool(flag.item())
    if args.e2e_steps > 0 and not fits:
        e2e = {"value": None, "unit": UNIT, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": 0,
               "skipped": "pinned host copies of the inputs (%.0f GB per rank) exceed 60%% of the"
                          " available host memory shared by this host's ranks" % (h2d / 1e9)}
    elif args.e2e_steps > 0:
        host = {}
        for k in names:
            host[k] = torch.empty(d[k].shape, dtype=d[k].dtype, pin_memory=True)
            host[k].copy_(d[k])
        loss_host = torch.empty(1, dtype=torch.float64, pin_memory=True)
        step.run_from_host(host, loss_host)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        kept_e, h2d_e, d2h_e = 0, 0, 0
        e0.record(stream)
        for _ in range(args.e2e_steps):
            hb, db = step.run_from_host(host, loss_host)
            h2d_e += hb
            d2h_e += db
            kept_e += step.T_kept
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms, kept_e = combine_ranks(e0.elapsed_time(e1), kept_e, world, dev)
        e2e = {"value": kept_e / (e_ms / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d_e // args.e2e_steps),
               "d2h_bytes_per_step": int(d2h_e // args.e2e_steps), "steps": args.e2e_steps,
               "host_inputs_bytes": int(h2d),
               "transfer": "selection inputs and per-token log-probs whole; logits of the kept "
                           "rollouts only (grpo_upload_kept), after the selection",
               "returned": "the loss (8 bytes) and the selection the host needs (kept counts, "
                           "kept per prompt, keep flags, kept offsets); logp and dlogits stay on "
                           "the device, where the backward pass consumes them"}
        del host

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        if args.loss == "gspo":
            cpu = cpu_baseline_gspo(w, b, step, d, args.cpu_seconds)
        else:
            cpu = cpu_baseline_ours(w, b, step, d, args.cpu_seconds)

    line = None
    if rank == 0:
        line = {
            "metric": METRIC, "value": r["value"], "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": elapsed_ms / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded; shapes and distributions of the paper's GRPO batches)",
            "config": dict(workload_desc(w, b["T"], step.T_kept, step.K), loss=args.loss),
            "gpu_launches": int(r["launches"]), "cuda_graph": r["use_graph"],
            "roofline": r["roofline"], "e2e": e2e,
            "cpu_baseline": cpu, "clocks": r["clocks"], "logp_fwd": logp_fwd, "lmhead": lmhead,
            "path_overhead": {"select_ms": select_ms,
                              "other_ms": elapsed_ms / K - select_ms - loss_ms,
                              "note": "select_ms: advantage, prune, compaction (and the kept-count"
                                      " read when host-synced), CUDA events; other_ms: the rest"
                                      " of the step (host ARS update, launch gaps)"},
            "loss_value": float(step.loss.item()), "ars_next_rollouts": step.n_next,
        }

    # the other full-size Qwen-vocabulary workloads, each in its own sub-record
    extra = [x for x in args.extra_configs.split(",") if x] if args.config in ("qwen", "2") else []
    if extra and args.prompts == 0 and args.group == 0:
        del r, b, d, step
        torch.cuda.empty_cache()
        configs = {}
        for name in extra:
            w2 = workloads.get(name)
            steps2 = max(1, int(round(args.extra_seconds * 1e3 / EXTRA_MS_GUESS.get(name, 20.0))))
            r2 = timed_steps(args, w2, rank_seed(args.seed, rank), world, local, dev, steps2,
                             args.warmup)
            configs[name] = sub_record(args, w2, r2, args.warmup)
            del r2
            torch.cuda.empty_cache()
        if line is not None:
            line["configs"] = configs
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
