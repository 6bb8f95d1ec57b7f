#!/usr/bin/env python3
"""Throughput of the DPB hot path on GB300: encode + decode + backward.

One step = dpb_encode, dpb_decode and dpb_backward over one batch of the
"wide" workload (T = 65536 tokens per GPU, d = 768, 2^20 features as 5 levels
of 16 children, beam 8, k = 64, bf16 storage with fp32 accumulation). Inputs
are synthetic: a planted tree of 64 parity directions per token plus
N(0, 0.1^2) noise, and grad_y ~ N(0, 1). The working set of a step (about
450 MB) is larger than the 129 MB L2, so no flush is needed between steps.

Prints one JSON line (rank 0). Under torchrun each rank runs its own token
shard (weak scaling, no data-path collective); the time is the max over
ranks. `--impl reference` times the CPU oracle on a bounded sample instead.
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "DPB tokens/sec (encode+decode+bwd) at d=768, 2^20 feats, 1 GB300; % of roofline"
WORKLOAD = "wide"
EMA_SAMPLE = 64        # rows per batch for the level >= 1 moments (§2.2 "Score Standardization")
EMA_ALPHA = 0.01       # EMA weight of one batch
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                  "sm_max_mhz": 2070.0}
GB300_SMS = 152
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e, nominal (the measured copy rate is the roofline's peak)
FP32_LANES_PER_SM = 128   # FADD/FFMA per SM per clock (measured; packed f32x2 gave no more)
INT_LOGIC_PER_SM = 64     # LOP3 per SM per clock (measured)
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic_wide_T65536.txt")
# files whose contents define each timed kernel (traffic figures are dropped
# when any of them changed after the counters were taken)
# the files holding each kernel's device code (host-side plan code does not
# change what a launch moves)
KERNEL_SOURCES = {
    "encode": ["dpb_encode_mma.cuh", "dpb_encode_mma.cu", "dpb_encode_mma_n2.cu", "dpb_select.cuh",
               "dpb_device.cuh"],
    "decode": ["dpb_decode.cu", "dpb_lut.cuh", "dpb_device.cuh"],
    "backward": ["dpb_backward.cu", "dpb_lut.cuh", "dpb_device.cuh"],
}


# ---------------------------------------------------------------------------
# distributed helpers (host logic; exercised by gloo tests on CPU)
# ---------------------------------------------------------------------------

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def shard_seed(base: int, rank: int) -> int:
    """Each rank draws its own token shard (weak scaling)."""
    return base + 1009 * rank


def max_over_ranks(value: float, world: int, device=None) -> float:
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def whole_job_rate(tokens_per_rank: int, world: int, steps: int, max_seconds: float) -> float:
    return tokens_per_rank * world * steps / max_seconds


# ---------------------------------------------------------------------------
# peaks, roofline and clocks
# ---------------------------------------------------------------------------

def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def sign_ops(signs: int, s: int) -> float:
    """Integer-logic operations that apply `signs` sign flips to stored
    elements of s bytes: a bf16 pair shares one 32-bit word, so one LOP3
    (XOR with the masked sign bits) flips two; an fp32 element takes one."""
    return signs / 2 if s == 2 else float(signs)


def algorithmic_work(cfg: dict, T: int, k_hash: float, s: int):
    """Per-launch algorithmic bytes and operations of each call (the method's
    own sums, not implementation overhead). s = bytes per stored element;
    k_hash = mean number of code entries that are hashed directions."""
    d, k, B = cfg["d"], cfg["k"], cfg["beam"]
    mma = sum(2 * B * cfg["children"][l] * d for l in range(1, cfg["levels"]))
    signs = (cfg["levels"] - 1) * B * d  # the x (.) phi~_p products of Eq. 6
    return {
        "encode": {"bytes": T * (d * s + 8 * k + 4), "tensor_flops": T * mma, "int_ops": T * sign_ops(signs, s)},
        "decode": {"bytes": T * (8 * k + 4 + d * s), "fp_ops": T * (k_hash * d + 3 * d)},
        "backward": {"bytes": T * (3 * d * s + 12 * k), "fp_ops": T * (2 * k_hash * d + 6 * d)},
    }


def alu_clock(peaks: dict, clocks: dict | None):
    """SM clock (MHz) for the ALU peaks: the median sampled while the kernels
    ran, else the maximum SM clock; and a note saying which."""
    if clocks and clocks.get("sm_mhz"):
        return float(clocks["sm_mhz"]), f"median SM clock sampled under load, {clocks['sm_mhz']:.0f} MHz"
    mhz = peaks.get("sm_max_mhz", 2070.0)
    return float(mhz), f"maximum SM clock {mhz:.0f} MHz (no clock samples)"


def peak_rates(peaks: dict, mhz: float | None = None):
    mhz = mhz or peaks.get("sm_max_mhz", 2070.0)
    return {"hbm": peaks["hbm_gbs"] * 1e9, "tensor": peaks["bf16_tflops_sustained"] * 1e12,
            "alu": GB300_SMS * FP32_LANES_PER_SM * mhz * 1e6, "int": GB300_SMS * INT_LOGIC_PER_SM * mhz * 1e6}


def roofline_for(name: str, work: dict, seconds: float, peaks: dict, src: str, traffic=None, clocks=None):
    """The slowest of the call's terms at peak (HBM bytes, tensor flops, FP32
    adds, integer logic ops) is its roofline; achieved = that term's work / time.
    The ALU peaks are taken at the SM clock sampled during the run."""
    mhz, clk_note = alu_clock(peaks, clocks)
    rate = peak_rates(peaks, mhz)
    keys = {"hbm": "bytes", "tensor": "tensor_flops", "alu": "fp_ops", "int": "int_ops"}
    terms = {b: work[kk] / rate[b] for b, kk in keys.items() if kk in work}
    bound = max(terms, key=terms.get)
    achieved = work[keys[bound]] / seconds
    if bound == "hbm":
        achieved, peak, unit = achieved / 1e9, peaks["hbm_gbs"], "GB/s"
        psrc = "copy"
    elif bound == "tensor":
        achieved, peak, unit = achieved / 1e12, peaks["bf16_tflops_sustained"], "TFLOP/s"
        psrc = "bf16 sustained"
    elif bound == "alu":
        achieved, peak, unit = achieved / 1e12, rate["alu"] / 1e12, "TFLOP/s"
        psrc = f"152 SMs x 128 FP32 adds/clock x {clk_note}"
    else:
        achieved, peak, unit = achieved / 1e12, rate["int"] / 1e12, "Tops/s"
        psrc = (f"152 SMs x 64 LOP3/clock x {clk_note}; one LOP3 flips the signs of a packed bf16 pair, "
                "so the work is half the sign applications")
    extra = {"frac_nominal": round(achieved / NOMINAL_HBM_GBS, 4)} if bound == "hbm" else {}
    # integer logic and FP32 adds are both plain ALU arithmetic ("alu"); "pipe"
    # says which of the two peaks the fraction is taken against
    return {**extra, "kernel": name, "bound": "alu" if bound == "int" else bound,
            "pipe": {"alu": "fp32", "int": "integer logic"}.get(bound),
            "achieved": round(achieved, 3), "peak": round(peak, 3),
            "unit": unit, "frac": round(achieved / peak, 4), "traffic": traffic,
            "algorithmic_bytes": int(work["bytes"]),
            "peak_source": f"{src} ({psrc})",
            "t_roofline_us": round(terms[bound] * 1e6, 2), "t_measured_us": round(seconds * 1e6, 2)}


def kernel_source_hash(name: str) -> str:
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[name]:
        with open(os.path.join(ROOT, "paper_2607_20652_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_traffic(name: str, T: int):
    """DRAM bytes per launch of `name` from the committed ncu figures, or None
    when absent, taken at another size, or the kernel changed since."""
    try:
        with open(TRAFFIC_FILE) as f:
            for line in f:
                parts = line.split()
                if len(parts) == 4 and not line.startswith("#") and parts[0] == name:
                    if int(parts[1]) == T and parts[3] == kernel_source_hash(name):
                        return int(parts[2])
    except (OSError, ValueError):
        pass
    return None


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled during the timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.gpu_id = gpu_id
        self.proc = None
        self.lines = []

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if self.gpu_id:
            cmd += ["-i", self.gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# workload
# ---------------------------------------------------------------------------

def workload_cfg():
    from paper_2607_20652_gb300 import configs
    return dict(configs.WORKLOADS[WORKLOAD])


def compose(tree, G, levels):
    """Feature indices of a planted tree through the plan's child map p ^ g_j."""
    nodes = [tree.roots.astype(np.int64)]
    for l in range(1, levels):
        par = np.take_along_axis(nodes[-1], tree.parent[l], axis=1)
        nodes.append(par ^ G[l][tree.gen[l]].astype(np.int64))
    return np.concatenate(nodes, axis=1).astype(np.int32)


def make_inputs_gpu(w, plan, seed, device):
    """Planted x (decoded by the library itself) + noise, and grad_y, on the GPU."""
    import torch
    from paper_2607_20652_gb300 import dpb, inputs
    T, d = w["T"], w["d"]
    _, G = plan.tables()
    tree = inputs.planted_tree(T, d, w["levels"], plan.config["children"], w["planted"], seed)
    idx_true = compose(tree, G, w["levels"])
    syn = dpb.Plan(d=d, levels=w["levels"], m_bits=w["m_bits"], children=w["children"],
                   beam=w["beam"], k=w["k"], dtype="f32", norm_match=0)
    y = dpb.decode(syn, torch.from_numpy(idx_true).to(device),
                   torch.from_numpy(tree.coef.astype(np.float32)).to(device))
    noise_h = inputs.normal((T, d), seed + 1000, w["noise"])
    x = (y + torch.from_numpy(noise_h).to(device)).to(torch.bfloat16).contiguous()
    gy_h = inputs.to_bf16(inputs.normal((T, d), seed + w["grad_seed"]))
    gy = torch.from_numpy(gy_h).to(device).to(torch.bfloat16)
    torch.cuda.synchronize(device)
    return x, gy, idx_true, {"tree": tree, "noise": noise_h, "gy": gy_h}


def oracle_sample(w, n_tokens, seed):
    """The same workload for the oracle: planted rows decoded by the oracle."""
    import oracle
    from paper_2607_20652_gb300 import inputs
    ref = oracle.resolve(d=w["d"], m_bits=w["m_bits"], levels=w["levels"], children=w["children"],
                         beam=w["beam"], k=w["k"])
    tree = inputs.planted_tree(n_tokens, w["d"], w["levels"], ref.children, w["planted"], seed)
    idx_true = compose(tree, ref.G, w["levels"])
    clean = oracle.decode(ref, idx_true, tree.coef, norm_match=0)
    x = inputs.to_bf16((clean + inputs.normal((n_tokens, w["d"]), seed + 1000, w["noise"])).astype(np.float32))
    gy = inputs.to_bf16(inputs.normal((n_tokens, w["d"]), seed + w["grad_seed"]))
    return ref, x.astype(np.float64), gy.astype(np.float64)


PARITY_ROWS = 256  # sampled tokens of the timed batch checked against the oracle


def parity_rows(w, host, T, seed):
    """Oracle leg, before timing: a seeded sample of rows of the timed batch
    and their x built by the oracle alone (its own generator table and decode
    of the planted code, plus the same noise), which then replace those rows
    on the GPU, so that no input of the check comes from the CUDA path."""
    import oracle
    from paper_2607_20652_gb300 import inputs
    ref = oracle.resolve(d=w["d"], m_bits=w["m_bits"], levels=w["levels"], children=w["children"],
                         beam=w["beam"], k=w["k"])
    rows = np.unique(np.concatenate([inputs.sample_rows(T, PARITY_ROWS, seed + 77), [0, T - 1]]))
    idx_true = compose(host["tree"], ref.G, w["levels"])[rows]
    clean = oracle.decode(ref, idx_true, host["tree"].coef[rows], norm_match=0)
    x_rows = inputs.to_bf16((clean + host["noise"][rows]).astype(np.float32))
    return ref, rows, x_rows


def parity_check(ref, rows, x_rows, gy_rows, out):
    """Oracle leg, after timing: the sampled rows' outputs of the last timed
    step against the oracle, by the rules of the -m gpu parity tests (codes as
    sets with near-ties counted, decode / r / gradients element by element on
    the GPU's own code)."""
    import oracle
    from tests import parity
    tol = parity.TOL["bf16"]
    xr = x_rows.astype(np.float64)
    gi, gvl, gxn = out["idx"], out["val"], out["xnorm"]
    res = {"tokens": int(len(rows)), "sample": f"{len(rows)} seeded rows of the timed batch (oracle-built x)",
           "rule": "indices as sets except near-ties (gap < 1e-5 relative, counted; their values checked against "
                   "their features' scores); val within 1e-5 |x|; "
                   "y, grad_x within 2e-2 max(|ref_i|, row rms) + 1 bf16 spacing, r and grad_val within 1e-5, "
                   "element by element, decode and backward on the GPU's own code"}
    try:
        idx_o, val_o, xn_o, gap = oracle.encode(ref, xr)
        parity.check_code_order(gi, gvl)
        near, worst_val = parity.compare_codes(gi, gvl, idx_o, val_o, gap, xn_o)
        parity.check_near_tie_values(ref, xr, gi, gvl, gap < parity.NEAR_TIE)
        res.update(near_ties=near, near_tie_tokens=[int(r) for r in np.asarray(rows)[gap < parity.NEAR_TIE]][:16],
                   val_err=worst_val)
        assert np.all(np.abs(gxn - xn_o) <= 1e-5 * np.maximum(xn_o, 1e-30)), "|x| differs"
        y_o = oracle.decode(ref, gi, gvl.astype(np.float64), gxn.astype(np.float64))
        res["y_err"] = parity.check_elementwise(out["y"], y_o, tol, True, "decode y")
        if out.get("r") is not None:
            r_o = oracle.decode(ref, gi, gvl.astype(np.float64), norm_match=0)
            res["r_err"] = parity.check_elementwise(out["r"], r_o, 1e-5, False, "kept r")
        gx_o, gv_o = oracle.backward(ref, xr, gi, gvl.astype(np.float64), gy_rows.astype(np.float64))
        res["gx_err"] = parity.check_elementwise(out["gx"], gx_o, tol, True, "grad_x")
        res["gv_err"] = parity.check_elementwise(out["gv"], gv_o, 1e-5, False, "grad_val")
        res["ok"] = True
    except AssertionError as e:
        res.update(ok=False, failure=str(e)[:300])
    for kk in ("val_err", "y_err", "r_err", "gx_err", "gv_err"):
        if kk in res:
            res[kk] = float(f"{res[kk]:.3e}")
    return res


def time_oracle(ref, x, gy):
    import oracle
    t0 = time.perf_counter()
    idx, val, xn, _ = oracle.encode(ref, x)
    oracle.decode(ref, idx, val, xn)
    oracle.backward(ref, x, idx, val, gy)
    return time.perf_counter() - t0


def host_cores() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def time_oracle_threads(ref, x, gy, threads: int):
    """The oracle over `threads` contiguous token ranges at once: each thread
    makes its own calls into the C oracle (which keeps no shared state;
    ctypes drops the GIL for the duration of each call)."""
    import concurrent.futures
    cuts = np.linspace(0, len(x), threads + 1).astype(int)
    t0 = time.perf_counter()
    with concurrent.futures.ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(lambda i: time_oracle(ref, x[cuts[i]:cuts[i + 1]], gy[cuts[i]:cuts[i + 1]]), range(threads)))
    return time.perf_counter() - t0


def cpu_baseline(w, budget_s: float, seed: int):
    """The oracle on the host cores: every core over a bounded sample (the
    line's value), and one core over a smaller one."""
    ref, x, gy = oracle_sample(w, 64, seed)
    per_tok = time_oracle(ref, x, gy) / 64
    n = int(max(64, min(16384, budget_s / 2 / max(per_tok, 1e-6))))
    cores = host_cores()
    n_all = int(max(n, min(16384, n * cores)))
    ref, x, gy = oracle_sample(w, n_all, seed)  # the single-thread run takes its first n
    secs = time_oracle(ref, x[:n], gy[:n])
    secs_all = time_oracle_threads(ref, x, gy, cores)
    return {"value": round(n_all / secs_all, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"first {n_all} tokens of the {WORKLOAD} workload (planted, seed {seed}); "
                      f"encode+decode+backward, C oracle (fp64) in {cores} threads over token ranges; "
                      f"{secs_all:.1f} s",
            "single_thread": {"value": round(n / secs, 2), "unit": "tokens/s", "cores": 1,
                              "sample": f"first {n} tokens, one thread; {secs:.1f} s"}}


# ---------------------------------------------------------------------------
# arms
# ---------------------------------------------------------------------------

def run_reference(args, world, rank):
    w = workload_cfg()
    if rank != 0:
        return 0
    n = args.ref_tokens
    cores = host_cores()
    ref, x, gy = oracle_sample(w, n, 0)
    for _ in range(args.warmup):
        time_oracle_threads(ref, x, gy, cores)
    times = [time_oracle_threads(ref, x, gy, cores) for _ in range(args.steps)]
    total = sum(times)
    value = n * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * total / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config_block(w, world),
        "cpu_baseline": {"kind": "oracle", "cores": cores, "value": round(value, 2), "unit": "tokens/s",
                         "sample": f"each step: the first {n} of the {w['T']} tokens of the {WORKLOAD} workload "
                                   f"(planted, seed 0), encode+decode+backward, C oracle (fp64) in {cores} "
                                   f"threads over token ranges"},
        "e2e": {"value": round(value, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def config_block(w, world, n_tokens=None, standardise=False):
    c = {"workload": WORKLOAD, "T_per_gpu": n_tokens or w["T"], "d": w["d"], "features": 2 ** w["m_bits"],
         "levels": w["levels"], "children": w["children"], "beam": w["beam"], "k": w["k"],
         "accumulate": "fp32", "inputs": "planted tree of 64 parity directions + N(0,0.1^2), bf16",
         "l2": "working set ~450 MB > 129 MB L2 (no flush needed)",
         "parallelism": f"dp{world} (independent token shards)"}
    if standardise:
        c["standardise"] = {"tables": "live fp32 mu/sigma (2^N each)", "ema_sample_rows": EMA_SAMPLE,
                            "ema_alpha": EMA_ALPHA,
                            "exchange": "all-reduce of the fp64 moment sums" if world > 1 else "none (1 rank)"}
    return c


def run_ours(args, world, rank, local):
    import torch
    from paper_2607_20652_gb300 import dpb

    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=device)
    w = workload_cfg()
    T, d = w["T"], w["d"]
    plan_kw = dict(d=d, levels=w["levels"], m_bits=w["m_bits"], children=w["children"],
                   beam=w["beam"], k=w["k"], dtype="bf16", norm_match=1)
    if args.coset:
        # the variant outside the paper: coset generators g0 ^ {0..15} per level,
        # scored by the Walsh-Hadamard path or by the contraction
        from paper_2607_20652_gb300 import inputs
        bits = dpb.Plan(**plan_kw).config["bits"]
        plan_kw.update(generators=inputs.coset_generators(bits, w["levels"], seed=5),
                       scoring=dpb.SCORING_COSET_WHT if args.coset == "wht" else dpb.SCORING_CONTRACTION)
    plan = dpb.Plan(**plan_kw)
    seed = shard_seed(w["seed"], rank)
    x, gy, idx_true, host = make_inputs_gpu(w, plan, seed, device)
    # oracle leg: seeded rows of the batch rebuilt by the oracle alone, checked after timing
    check = rank == 0 and world == 1 and not args.no_parity and not args.standardise and not args.coset
    if check:
        pref, prows, px = parity_rows(w, host, T, seed)
        x[torch.from_numpy(prows).to(device)] = torch.from_numpy(px).to(device).to(torch.bfloat16)
        pgy = host["gy"][prows]
    del host
    k = plan.code_len
    idx = torch.empty((T, k), dtype=torch.int32, device=device)
    val = torch.empty((T, k), dtype=torch.float32, device=device)
    xn = torch.empty((T,), dtype=torch.float32, device=device)
    y = torch.empty_like(x)
    gx = torch.empty_like(x)
    gv = torch.empty((T, k), dtype=torch.float32, device=device)
    # decode keeps r (fp32) for the backward, which then does not rebuild it
    rk = None if args.no_keep_r else torch.empty((T, d), dtype=torch.float32, device=device)
    ws = plan.workspace(T, device)
    stream = torch.cuda.current_stream(device)
    # live standardisation (§2.2): encode and backward read the tables, and
    # each step ends with the EMA update from the level-0 column sums and a
    # 64-row sub-sample (tables start at mu = 0, sigma = 1)
    std = args.standardise
    mu_t = sg_t = acc = None
    samples = []
    if std:
        mu_t = torch.zeros(plan.n_features, dtype=torch.float32, device=device)
        sg_t = torch.ones(plan.n_features, dtype=torch.float32, device=device)
        acc = dpb.stats_buffer(plan, device)
        gen = torch.Generator().manual_seed(seed)
        samples = [dpb.sample_rows(T, EMA_SAMPLE, gen, device) for _ in range(max(args.steps, args.warmup))]
    stages = ["encode", "decode", "backward"] + (["stats"] if std else [])

    def step(ev=None, i=0):
        if ev:
            ev[0].record(stream)
        dpb.encode(plan, x, mu_t, sg_t, idx=idx, val=val, xnorm=xn, workspace=ws, stream=stream)
        if ev:
            ev[1].record(stream)
        dpb.decode(plan, idx, val, xn, y=y, workspace=ws, stream=stream, r_out=rk)
        if ev:
            ev[2].record(stream)
        dpb.backward(plan, x, idx, val, gy, sigma=sg_t, grad_x=gx, grad_val=gv, workspace=ws, stream=stream, r=rk)
        if ev:
            ev[3].record(stream)
        if std:
            dpb.stats_step(plan, x, mu_t, sg_t, EMA_ALPHA, samples[i % len(samples)], acc=acc, workspace=ws,
                           stream=stream)
            if ev:
                ev[4].record(stream)

    for i in range(args.warmup):
        step(None, i)
    torch.cuda.synchronize(device)
    status = dpb.workspace_status(ws)

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)] for _ in range(args.steps)]
    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
    except Exception:
        gpu_id = None
    clocks = ClockSampler(gpu_id)
    clocks.start()
    time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize(device)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for i in range(args.steps):
        step(evs[i], i)
    end.record(stream)
    torch.cuda.synchronize(device)
    barrier(world)
    ms = start.elapsed_time(end)
    # A timed region shorter than the clock window is followed by the same
    # step for the rest of the window, so that the sampler (200 ms period)
    # sees the clock these kernels run at; its per-kernel times are reported
    # beside the timed ones.
    sustained = None
    if ms < 1e3 * args.clock_seconds:
        n_more = max(1, int((1e3 * args.clock_seconds - ms) / max(ms / args.steps, 1e-3)))
        sev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)] for _ in range(n_more)]
        for i in range(n_more):
            step(sev[i], args.steps + i)
        torch.cuda.synchronize(device)
        sustained = {"steps": n_more, "ms_per_step": round(sum(e[0].elapsed_time(e[-1]) for e in sev) / n_more, 4),
                     "kernels_ms": {n: round(statistics.mean(e[j].elapsed_time(e[j + 1]) for e in sev), 4)
                                    for j, n in enumerate(stages)}}
    clk = clocks.stop()
    clk["window"] = ("the timed steps" if sustained is None else
                     f"the timed steps and {sustained['steps']} more of the same step right after "
                     f"({args.clock_seconds:.1f} s in all)")
    ms_max = max_over_ranks(ms, world, device)
    kern_ms = {n: statistics.mean(e[j].elapsed_time(e[j + 1]) for e in evs) for j, n in enumerate(stages)}
    if std:
        status |= dpb.workspace_status(ws)

    # algorithmic work and roofline of the dominant kernel
    idx_np = idx.cpu().numpy()
    k_hash = float(np.mean(np.sum(idx_np >= d, axis=1)))
    recovered = float(np.mean([len(set(idx_np[t]) & set(idx_true[t])) / k for t in range(0, T, 64)]))
    peaks, src = load_peaks()
    work = algorithmic_work(plan.config, T, k_hash, 2)
    if std:
        # the column pass reads x once; the update scans the 2^N counts
        work["stats"] = {"bytes": T * d * 2 + 8 * plan.n_features}
    dom = max(kern_ms, key=kern_ms.get)
    roof = roofline_for(dom, work[dom], kern_ms[dom] / 1e3, peaks, src, measured_traffic(dom, T), clocks=clk)
    kernels = {n: {"ms": round(v, 4), **{kk: vv for kk, vv in
                                         roofline_for(n, work[n], v / 1e3, peaks, src, clocks=clk).items()
                                         if kk in ("bound", "pipe", "frac", "t_roofline_us")}}
               for n, v in kern_ms.items()}
    step_roof_us = sum(kernels[n]["t_roofline_us"] for n in kernels)

    par = None
    if check:
        pr = torch.from_numpy(prows).to(device)
        out = {"idx": idx[pr].cpu().numpy(), "val": val[pr].cpu().numpy(), "xnorm": xn[pr].cpu().numpy(),
               "y": y[pr].float().cpu().numpy(), "gx": gx[pr].float().cpu().numpy(), "gv": gv[pr].cpu().numpy(),
               "r": None if rk is None else rk[pr].cpu().numpy()}
        par = parity_check(pref, prows, px, pgy, out)

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e and not std:
        e2e = run_e2e(plan, x, gy, args, device, stream, world)

    value = whole_job_rate(T, world, args.steps, ms_max / 1e3)
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic", "config": {**config_block(w, world, standardise=std),
                                         **({"generators": "coset g0 ^ {0..15} per level (variant outside the paper)",
                                             "scoring": args.coset} if args.coset else {})},
        "roofline": roof,
        "step_roofline": {"t_roofline_us": round(step_roof_us, 2),
                          "t_measured_us": round(1e3 * ms_max / args.steps, 2),
                          "frac": round(step_roof_us / (1e3 * ms_max / args.steps), 4)},
        "kernels": kernels, "k_hash": round(k_hash, 2), "planted_recovery": round(recovered, 4),
        "r_kept": rk is not None,
        "gpu_launches": (3 + (3 if std else 0)) * args.steps, "clocks": clk, "device_status": status,
    }
    if sustained:
        line["sustained"] = sustained
    if par is not None:
        line["parity"] = par
    if e2e:
        line["e2e"] = e2e
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds, 0)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def run_e2e(plan, x, gy, args, device, stream, world):
    """The metric through the public calls with host buffers: every step copies
    its inputs from pinned host memory and its outputs back, inside the timed
    region. The batch runs as chunks on a few streams, so one chunk's copies
    overlap another's kernels (each stream keeps its own device buffers and
    workspace; calls on one stream run in order). A chunk's x and grad_y sit
    side by side in host memory and move in one copy; its outputs come back in
    two (the [C, k] arrays, then y and grad_x)."""
    import torch
    from paper_2607_20652_gb300 import dpb
    T, d = x.shape
    k = plan.code_len
    nch = max(1, args.e2e_chunks)
    while T % nch:
        nch -= 1
    C = T // nch
    hin = torch.empty((nch, 2, C, d), dtype=x.dtype).pin_memory()       # [chunk][x | grad_y]
    hin[:, 0].copy_(x.view(nch, C, d))
    hin[:, 1].copy_(gy.view(nch, C, d))
    hsmall = torch.empty((nch, 3, C, k), dtype=torch.int32).pin_memory()  # [chunk][idx | val | grad_val]
    hbig = torch.empty((nch, 2, C, d), dtype=x.dtype).pin_memory()       # [chunk][y | grad_x]
    nstreams = max(1, min(args.e2e_streams, nch))
    streams = [torch.cuda.Stream(device) for _ in range(nstreams)]
    bufs = []
    for _ in range(nstreams):
        inp = torch.empty((2, C, d), dtype=x.dtype, device=device)
        small = torch.empty((3, C, k), dtype=torch.int32, device=device)
        big = torch.empty((2, C, d), dtype=x.dtype, device=device)
        bufs.append({"inp": inp, "x": inp[0], "gy": inp[1], "small": small, "idx": small[0],
                     "val": small[1].view(torch.float32), "gv": small[2].view(torch.float32),
                     "big": big, "y": big[0], "gx": big[1],
                     "xn": torch.empty((C,), dtype=torch.float32, device=device),
                     "r": None if args.no_keep_r else torch.empty((C, d), dtype=torch.float32, device=device),
                     "ws": plan.workspace(C, device)})

    def step():
        for i in range(nch):
            st, b = streams[i % nstreams], bufs[i % nstreams]
            with torch.cuda.stream(st):
                b["inp"].copy_(hin[i], non_blocking=True)
                dpb.encode(plan, b["x"], idx=b["idx"], val=b["val"], xnorm=b["xn"], workspace=b["ws"], stream=st)
                dpb.decode(plan, b["idx"], b["val"], b["xn"], y=b["y"], workspace=b["ws"], stream=st, r_out=b["r"])
                dpb.backward(plan, b["x"], b["idx"], b["val"], b["gy"], grad_x=b["gx"], grad_val=b["gv"],
                             workspace=b["ws"], stream=st, r=b["r"])
                hsmall[i].copy_(b["small"], non_blocking=True)
                hbig[i].copy_(b["big"], non_blocking=True)

    def timed(fn):
        for _ in range(max(1, args.warmup)):
            fn()
        torch.cuda.synchronize(device)
        n = max(3, min(args.steps // 2, 400))
        barrier(world)
        t0 = time.perf_counter()
        for _ in range(n):
            fn()
        torch.cuda.synchronize(device)
        return n, max_over_ranks(time.perf_counter() - t0, world, device)

    steps, secs = timed(step)
    status = 0
    for b in bufs:
        status |= dpb.workspace_status(b["ws"])
    bi = hin.numel() * hin.element_size()
    bo = hsmall.numel() * hsmall.element_size() + hbig.numel() * hbig.element_size()
    return {"value": round(whole_job_rate(T, world, steps, secs), 1), "unit": "tokens/s",
            "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo, "steps": steps,
            "chunks": nch, "streams": nstreams, "device_status": status}


# ---------------------------------------------------------------------------
# the small global-mode workloads (supplementary lines; they fit in L2)
# ---------------------------------------------------------------------------

L2_FLUSH_BYTES = 512 << 20  # written between steps: more than the 129 MB L2


def run_global_small(args, world, rank, local):
    """The tiny (fp32, encode + decode + backward) and GPT-2-width (bf16 with 5%
    outlier rows, encode + decode) workloads. Their working sets fit in L2, so
    every step is timed on its own (CUDA events around its calls) after a
    512 MB write that flushes L2; the line's time is the mean of those steps.
    A seeded sample of rows (every row of tiny) is checked against the oracle
    on the last step's outputs."""
    import torch
    from paper_2607_20652_gb300 import configs, dpb, inputs
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    w = dict(configs.WORKLOADS[args.workload])
    T, d = w["T"], w["d"]
    bwd = w["passes"] == "fwd+bwd"
    plan = dpb.Plan(d=d, levels=w["levels"], m_bits=w["m_bits"], children=w["children"], beam=w["beam"],
                    k=w["k"], dtype=w["dtype"], norm_match=1)
    seed = shard_seed(w["seed"], rank)
    xh = inputs.gaussian_rows(T, d, seed, w.get("outlier_frac", 0.0), w.get("outlier_scale", 10.0))
    gyh = inputs.normal((T, d), seed + w.get("grad_seed", 1))
    if w["dtype"] == "bf16":
        xh, gyh = inputs.to_bf16(xh), inputs.to_bf16(gyh)
    x = torch.from_numpy(xh).to(device).to(plan.torch_dtype)
    gy = torch.from_numpy(gyh).to(device).to(plan.torch_dtype)
    k = plan.code_len
    idx = torch.empty((T, k), dtype=torch.int32, device=device)
    val = torch.empty((T, k), dtype=torch.float32, device=device)
    xn = torch.empty((T,), dtype=torch.float32, device=device)
    y, gx = torch.empty_like(x), torch.empty_like(x)
    gv = torch.empty((T, k), dtype=torch.float32, device=device)
    rk = torch.empty((T, d), dtype=torch.float32, device=device) if bwd else None
    ws = plan.workspace(T, device)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
    stream = torch.cuda.current_stream(device)
    stages = ["encode", "decode"] + (["backward"] if bwd else [])

    def step(ev=None):
        flush.fill_(1.0)
        if ev:
            ev[0].record(stream)
        dpb.encode(plan, x, idx=idx, val=val, xnorm=xn, workspace=ws, stream=stream)
        if ev:
            ev[1].record(stream)
        dpb.decode(plan, idx, val, xn, y=y, workspace=ws, stream=stream, r_out=rk)
        if ev:
            ev[2].record(stream)
        if bwd:
            dpb.backward(plan, x, idx, val, gy, grad_x=gx, grad_val=gv, workspace=ws, stream=stream, r=rk)
            if ev:
                ev[3].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(device)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)] for _ in range(args.steps)]
    clocks = ClockSampler(None)
    clocks.start()
    time.sleep(0.3)
    barrier(world)
    for e in evs:
        step(e)
    torch.cuda.synchronize(device)
    barrier(world)
    clk = clocks.stop()
    ms = statistics.mean(e[0].elapsed_time(e[-1]) for e in evs)
    ms_max = max_over_ranks(ms, world, device)
    kern_ms = {n: statistics.mean(e[j].elapsed_time(e[j + 1]) for e in evs) for j, n in enumerate(stages)}
    idx_np = idx.cpu().numpy()
    k_hash = float(np.mean(np.sum(idx_np >= d, axis=1)))
    peaks, src = load_peaks()
    s_el = 4 if w["dtype"] == "f32" else 2
    work = algorithmic_work(plan.config, T, k_hash, s_el)
    kernels = {n: {"ms": round(v, 4), **{kk: vv for kk, vv in
                                         roofline_for(n, work[n], v / 1e3, peaks, src, clocks=clk).items()
                                         if kk in ("bound", "pipe", "frac", "t_roofline_us")}}
               for n, v in kern_ms.items()}
    step_roof_us = sum(kernels[n]["t_roofline_us"] for n in kernels)
    dom = max(kern_ms, key=kern_ms.get)
    line = {
        "metric": f"DPB tokens/sec ({'+'.join(stages)}), {args.workload} config, 1 GB300",
        "value": round(whole_job_rate(T, world, 1, ms_max / 1e3), 1), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_max, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w["dtype"], "data": "synthetic",
        "config": {"workload": args.workload, "T_per_gpu": T, "d": d, "features": 2 ** w["m_bits"],
                   "levels": w["levels"], "children": w["children"], "beam": w["beam"], "k": w["k"],
                   "inputs": "x ~ N(0,1)" + (f", {int(100 * w['outlier_frac'])}% of rows x{w['outlier_scale']:g}"
                                             if w.get("outlier_frac") else "") + f", {w['dtype']}",
                   "l2": "512 MB written before every step (flush); each step timed on its own"},
        "roofline": roofline_for(dom, work[dom], kern_ms[dom] / 1e3, peaks, src, clocks=clk),
        "step_roofline": {"t_roofline_us": round(step_roof_us, 2), "t_measured_us": round(1e3 * ms_max, 2),
                          "frac": round(step_roof_us / (1e3 * ms_max), 4)},
        "kernels": kernels, "k_hash": round(k_hash, 2), "gpu_launches": len(stages) * args.steps, "clocks": clk,
        "device_status": dpb.workspace_status(ws),
    }
    if rank == 0 and world == 1 and not args.no_parity:
        line["parity"] = small_parity(w, plan, xh, gyh if bwd else None,
                                      {"idx": idx, "val": val, "xnorm": xn, "y": y, "gx": gx if bwd else None,
                                       "gv": gv if bwd else None, "r": rk})
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = small_cpu_baseline(w, xh, gyh if bwd else None, plan)
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def _small_ref(w, plan):
    import oracle
    c = plan.config
    return oracle.resolve(d=c["d"], m_bits=w["m_bits"], levels=c["levels"], children=c["children"],
                          beam=c["beam"], k=c["k"], seed=c["generator_seed"], norm_match=c["norm_match"],
                          t=c["field_t"], poly=c["field_poly"], bits=c["bits"])


def small_parity(w, plan, xh, gyh, out):
    """Oracle leg: every row of tiny, 256 seeded rows of GPT-2 width, checked
    by the rules of the -m gpu parity tests."""
    import oracle
    from paper_2607_20652_gb300 import inputs
    from tests import parity
    T = len(xh)
    rows = np.arange(T) if T <= 256 else np.unique(np.concatenate([inputs.sample_rows(T, 256, 77), [0, T - 1]]))
    ref = _small_ref(w, plan)
    bf16 = w["dtype"] == "bf16"
    tol = parity.TOL["bf16" if bf16 else "f32"]
    import torch

    def host(v):
        if v is None:
            return None
        return (v.cpu().numpy() if v.dtype == torch.int32 else v.float().cpu().numpy())[rows]

    get = {kk: host(v) for kk, v in out.items()}
    xr = xh[rows].astype(np.float64)
    res = {"tokens": int(len(rows)), "sample": "every row" if T <= 256 else f"{len(rows)} seeded rows"}
    try:
        idx_o, val_o, xn_o, gap = oracle.encode(ref, xr)
        parity.check_code_order(get["idx"], get["val"])
        near, worst = parity.compare_codes(get["idx"], get["val"], idx_o, val_o, gap, xn_o)
        parity.check_near_tie_values(ref, xr, get["idx"], get["val"], gap < parity.NEAR_TIE)
        res.update(near_ties=near, val_err=worst)
        y_o = oracle.decode(ref, get["idx"], get["val"].astype(np.float64), get["xnorm"].astype(np.float64))
        res["y_err"] = parity.check_elementwise(get["y"], y_o, tol, bf16, "decode y")
        if gyh is not None:
            r_o = oracle.decode(ref, get["idx"], get["val"].astype(np.float64), norm_match=0)
            res["r_err"] = parity.check_elementwise(get["r"], r_o, 1e-5, False, "kept r")
            gx_o, gv_o = oracle.backward(ref, xr, get["idx"], get["val"].astype(np.float64),
                                         gyh[rows].astype(np.float64))
            res["gx_err"] = parity.check_elementwise(get["gx"], gx_o, tol, bf16, "grad_x")
            res["gv_err"] = parity.check_elementwise(get["gv"], gv_o, 1e-5, False, "grad_val")
        res["ok"] = True
    except AssertionError as e:
        res.update(ok=False, failure=str(e)[:300])
    for kk in ("val_err", "y_err", "r_err", "gx_err", "gv_err"):
        if kk in res:
            res[kk] = float(f"{res[kk]:.3e}")
    return res


def small_cpu_baseline(w, xh, gyh, plan):
    """The oracle on the host cores over the same rows (all of tiny; the first
    2048 of GPT-2 width), as for the wide workload."""
    import oracle
    ref = _small_ref(w, plan)
    n = min(len(xh), 2048)
    x = xh[:n].astype(np.float64)
    cores = host_cores()
    cuts = np.linspace(0, n, cores + 1).astype(int)

    def part(i):
        xs = x[cuts[i]:cuts[i + 1]]
        idx, val, xn, _ = oracle.encode(ref, xs)
        oracle.decode(ref, idx, val, xn)
        if gyh is not None:
            oracle.backward(ref, xs, idx, val, gyh[cuts[i]:cuts[i + 1]].astype(np.float64))

    import concurrent.futures
    t0 = time.perf_counter()
    with concurrent.futures.ThreadPoolExecutor(max_workers=cores) as ex:
        list(ex.map(part, range(cores)))
    secs = time.perf_counter() - t0
    return {"value": round(n / secs, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"first {n} tokens of the {'tiny' if len(xh) <= 256 else 'gpt2'} workload, "
                      f"C oracle (fp64) in {cores} threads over token ranges; {secs:.2f} s"}


# ---------------------------------------------------------------------------
# the paper's per-level layouts (supplementary lines; the headline is "wide")
# ---------------------------------------------------------------------------

def per_level_work(w, T: int, k_hash: float, s: int):
    """Algorithmic work of the per-level layouts: level l scores K_{l-1} x
    Delta_l children (Eq. 6: 2 d flops and d sign applications each)."""
    d, kl, ch = w["d"], w["k_per_level"], w["children"]
    code = sum(kl)
    mma = sum(2 * kl[l - 1] * ch[l] * d for l in range(1, w["levels"]))
    signs = sum(kl[l - 1] * d for l in range(1, w["levels"]))
    return {
        "encode": {"bytes": T * (d * s + 8 * code + 4), "tensor_flops": T * mma, "int_ops": T * sign_ops(signs, s)},
        "decode": {"bytes": T * (8 * code + 4 + d * s), "fp_ops": T * (k_hash * d + 3 * d)},
        "backward": {"bytes": T * (3 * d * s + 12 * code), "fp_ops": T * (2 * k_hash * d + 6 * d)},
    }


def run_per_level(args, world, rank, local):
    import torch
    from paper_2607_20652_gb300 import configs, dpb, inputs

    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    w = dict(configs.PER_LEVEL[args.workload])
    T, d = w["T"], w["d"]
    plan = dpb.Plan(d=d, levels=w["levels"], bits=w["bits"], children=w["children"], dtype="bf16",
                    select_mode=dpb.SELECT_PER_LEVEL, k_per_level=w["k_per_level"])
    seed = shard_seed(w["seed"], rank)
    x = torch.from_numpy(inputs.to_bf16(inputs.gaussian_rows(T, d, seed))).to(device).to(torch.bfloat16)
    gy = torch.from_numpy(inputs.to_bf16(inputs.normal((T, d), seed + w["grad_seed"]))).to(device).to(torch.bfloat16)
    k = plan.code_len
    idx = torch.empty((T, k), dtype=torch.int32, device=device)
    val = torch.empty((T, k), dtype=torch.float32, device=device)
    xn = torch.empty((T,), dtype=torch.float32, device=device)
    y, gx = torch.empty_like(x), torch.empty_like(x)
    gv = torch.empty((T, k), dtype=torch.float32, device=device)
    ws = plan.workspace(T, device)
    stream = torch.cuda.current_stream(device)
    std = args.standardise
    mu_t = sg_t = acc = None
    samples = []
    if std:
        mu_t = torch.zeros(plan.n_features, dtype=torch.float32, device=device)
        sg_t = torch.ones(plan.n_features, dtype=torch.float32, device=device)
        acc = dpb.stats_buffer(plan, device)
        gen = torch.Generator().manual_seed(seed)
        samples = [dpb.sample_rows(T, EMA_SAMPLE, gen, device) for _ in range(max(args.steps, args.warmup))]
    stages = ["encode", "decode", "backward"] + (["stats"] if std else [])

    def step(ev=None, i=0):
        if ev:
            ev[0].record(stream)
        dpb.encode(plan, x, mu_t, sg_t, idx=idx, val=val, xnorm=xn, workspace=ws, stream=stream)
        if ev:
            ev[1].record(stream)
        dpb.decode(plan, idx, val, xn, y=y, workspace=ws, stream=stream)
        if ev:
            ev[2].record(stream)
        dpb.backward(plan, x, idx, val, gy, sigma=sg_t, grad_x=gx, grad_val=gv, workspace=ws, stream=stream)
        if ev:
            ev[3].record(stream)
        if std:
            dpb.stats_step(plan, x, mu_t, sg_t, EMA_ALPHA, samples[i], acc=acc, workspace=ws, stream=stream)
            if ev:
                ev[4].record(stream)

    for i in range(args.warmup):
        step(None, i)
    torch.cuda.synchronize(device)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)] for _ in range(args.steps)]
    clocks = ClockSampler(None)
    clocks.start()
    time.sleep(0.3)
    barrier(world)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for i in range(args.steps):
        step(evs[i], i)
    end.record(stream)
    torch.cuda.synchronize(device)
    barrier(world)
    clk = clocks.stop()
    ms_max = max_over_ranks(start.elapsed_time(end), world, device)
    kern_ms = {n: statistics.mean(e[j].elapsed_time(e[j + 1]) for e in evs) for j, n in enumerate(stages)}
    k_hash = float(np.mean(np.sum(idx.cpu().numpy() >= d, axis=1)))
    peaks, src = load_peaks()
    work = per_level_work(w, T, k_hash, 2)
    if std:
        work["stats"] = {"bytes": T * d * 2 + 8 * plan.n_features}
    kernels = {n: {"ms": round(v, 4), **{kk: vv for kk, vv in
                                         roofline_for(n, work[n], v / 1e3, peaks, src, clocks=clk).items()
                                         if kk in ("bound", "pipe", "frac", "t_roofline_us", "achieved", "unit")}}
               for n, v in kern_ms.items()}
    dom = max(kern_ms, key=kern_ms.get)
    line = {
        "metric": f"DPB tokens/sec (encode+decode+bwd), per-level selection, paper {args.workload[5:].upper()} layout "
                  f"(d={d}, K={w['k_per_level']}, Delta=256), 1 GB300",
        "value": round(whole_job_rate(T, world, args.steps, ms_max / 1e3), 1), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_max / args.steps, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": args.workload, "T_per_gpu": T, "d": d, "levels": w["levels"], "bits": w["bits"],
                   "children": w["children"], "k_per_level": w["k_per_level"], "select": "per_level",
                   "inputs": "bf16 x ~ N(0,1), grad_y ~ N(0,1)",
                   "l2": "inputs (2 x 128 MiB) larger than the 129 MB L2 (no flush needed)",
                   **({"standardise": {"tables": "live fp32 mu/sigma (2^N each)", "ema_sample_rows": EMA_SAMPLE,
                                       "ema_alpha": EMA_ALPHA}} if std else {})},
        "roofline": roofline_for(dom, work[dom], kern_ms[dom] / 1e3, peaks, src, clocks=clk),
        "kernels": kernels, "k_hash": round(k_hash, 2), "gpu_launches": (3 + (3 if std else 0)) * args.steps,
        "clocks": clk,
        "device_status": dpb.workspace_status(ws),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------
# the sweep at d = 768, T = 32768: tokens/s and roofline fraction per point
# ---------------------------------------------------------------------------

def run_sweep(args, world, rank, local):
    import torch
    from paper_2607_20652_gb300 import configs, dpb

    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    stream = torch.cuda.current_stream(device)
    peaks, src = load_peaks()
    points = []
    steps = max(3, args.steps // 4)
    clocks = ClockSampler(None)
    clocks.start()
    for w in configs.SWEEP:
        T, d = w["T"], w["d"]
        plan = dpb.Plan(d=d, levels=w["levels"], m_bits=w["m_bits"], children=w["children"], beam=w["beam"],
                        k=w["k"], dtype="bf16")
        g = torch.Generator(device=device).manual_seed(shard_seed(w["seed"], rank) + w["m_bits"] * 100 + w["k"])
        x = torch.randn((T, d), generator=g, device=device).to(torch.bfloat16)
        gy = torch.randn((T, d), generator=g, device=device).to(torch.bfloat16)
        k = plan.code_len
        idx = torch.empty((T, k), dtype=torch.int32, device=device)
        val = torch.empty((T, k), dtype=torch.float32, device=device)
        xn = torch.empty((T,), dtype=torch.float32, device=device)
        y, gx = torch.empty_like(x), torch.empty_like(x)
        gv = torch.empty((T, k), dtype=torch.float32, device=device)
        rk = torch.empty((T, d), dtype=torch.float32, device=device)
        ws = plan.workspace(T, device)

        def step(ev=None):
            if ev:
                ev[0].record(stream)
            dpb.encode(plan, x, idx=idx, val=val, xnorm=xn, workspace=ws, stream=stream)
            if ev:
                ev[1].record(stream)
            dpb.decode(plan, idx, val, xn, y=y, workspace=ws, stream=stream, r_out=rk)
            if ev:
                ev[2].record(stream)
            dpb.backward(plan, x, idx, val, gy, grad_x=gx, grad_val=gv, workspace=ws, stream=stream, r=rk)
            if ev:
                ev[3].record(stream)

        for _ in range(2):
            step()
        torch.cuda.synchronize(device)
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
        barrier(world)
        for e in evs:
            step(e)
        torch.cuda.synchronize(device)
        kern = {n: statistics.mean(e[j].elapsed_time(e[j + 1]) for e in evs)
                for j, n in enumerate(("encode", "decode", "backward"))}
        ms = max_over_ranks(sum(kern.values()), world, device)
        k_hash = float(np.mean(np.sum(idx.cpu().numpy() >= d, axis=1)))
        work = algorithmic_work(plan.config, T, k_hash, 2)
        points.append({"features": 2 ** w["m_bits"], "k": w["k"], "beam": w["beam"],
                       "encoder": "tensor-core" if w["beam"] <= 16 else "general",
                       "tokens_per_s": round(whole_job_rate(T, world, 1, ms / 1e3), 1),
                       "ms": {n: round(v, 4) for n, v in kern.items()},
                       "_work": work, "_kern": kern, "_ms": ms,
                       "device_status": dpb.workspace_status(ws)})
        del x, gy, idx, val, xn, y, gx, gv, rk, ws, plan
        torch.cuda.empty_cache()
    clk = clocks.stop()
    for pt in points:
        work, kern, ms = pt.pop("_work"), pt.pop("_kern"), pt.pop("_ms")
        roofs = {n: roofline_for(n, work[n], kern[n] / 1e3, peaks, src, clocks=clk) for n in kern}
        pt["frac"] = {n: r["frac"] for n, r in roofs.items()}
        pt["step_roofline_frac"] = round(sum(r["t_roofline_us"] for r in roofs.values()) / (1e3 * ms), 4)
    line = {"metric": "DPB sweep at d=768, T=32768: tokens/s (encode+decode+bwd) and roofline fraction per point",
            "unit": "tokens/s", "n_gpus": world, "steps": steps, "warmup": 2, "higher_is_better": True,
            "scaling": "weak", "dtype": "bf16", "data": "synthetic (x, grad_y ~ N(0, 1), bf16)",
            "config": {"workload": "sweep", "T_per_gpu": 32768, "d": 768, "levels": 5, "children": 16,
                       "r_kept": "decode keeps r (fp32) for the backward"},
            "clocks": clk, "points": points}
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------
# the ParityTransformer step (GPT-2 small shape): the DPB's share of a step
# ---------------------------------------------------------------------------

GPT2_SMALL = dict(layers=12, d=768, heads=12, d_mlp=3072, vocab=50257, context=1024, batch=8)
GPT2_DPB = dict(levels=5, m_bits=20, children=16, beam=8, k=64)


def run_transformer(args, world, rank, local):
    import torch
    from paper_2607_20652_gb300 import transformer

    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    c = GPT2_SMALL
    B, S = c["batch"], c["context"]
    g = torch.Generator().manual_seed(shard_seed(7, rank))
    ids = torch.randint(0, c["vocab"], (B, S), generator=g).to(device)
    tgt = torch.randint(0, c["vocab"], (B, S), generator=g).to(device)
    dpb_kw = dict(GPT2_DPB, ema=EMA_ALPHA if args.standardise else None)

    def build(with_dpb):
        torch.manual_seed(0)
        m = transformer.ParityTransformer(layers=c["layers"], d=c["d"], heads=c["heads"], d_mlp=c["d_mlp"],
                                          vocab=c["vocab"], context=c["context"],
                                          dpb=dpb_kw if with_dpb else None, device=device)
        return m, torch.optim.AdamW(m.parameters(), lr=1e-4, fused=True)

    def measure(model, opt, dpbs):
        stream = torch.cuda.current_stream(device)

        def step():
            opt.zero_grad(set_to_none=True)
            loss = model(ids, tgt)
            loss.backward()
            opt.step()
            return loss

        for _ in range(args.warmup):
            step()
        torch.cuda.synchronize(device)
        for layer in dpbs:
            layer.timing = []
        barrier(world)
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for _ in range(args.steps):
            loss = step()
        end.record(stream)
        torch.cuda.synchronize(device)
        ms = max_over_ranks(start.elapsed_time(end), world, device) / args.steps
        parts = {"forward": 0.0, "backward": 0.0}
        for layer in dpbs:
            for which, ev in layer.timing:
                parts[which] += ev[0].elapsed_time(ev[1]) / args.steps
            layer.timing = None
        return ms, parts, float(loss.detach())

    model, opt = build(True)
    ms, parts, loss = measure(model, opt, model.dpb_layers())
    status = 0
    from paper_2607_20652_gb300 import dpb as _dpb
    for layer in model.dpb_layers():
        status |= _dpb.workspace_status(layer._ws)
    del model, opt
    torch.cuda.empty_cache()
    dense_ms = None
    if not args.no_dense:
        dense, dopt = build(False)
        dense_ms, _, _ = measure(dense, dopt, [])
        del dense, dopt
    tokens = B * S
    dpb_ms = parts["forward"] + parts["backward"]
    per_layer = (3 + (4 if args.standardise else 0))
    line = {
        "metric": "ParityTransformer GPT-2-small training step (fwd + bwd + AdamW), tokens/s; DPB share of the step",
        "value": round(whole_job_rate(tokens, world, 1, ms / 1e3), 1), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic (uniform random token ids)",
        "config": {"workload": "gpt2small", **c, "tokens_per_step": tokens,
                   "dpb": {**GPT2_DPB, "placement": "before every MLP input (§3)",
                           "standardise": bool(args.standardise)},
                   "weights": "random init (std 0.02), bf16; AdamW fused", "parallelism": f"dp{world}"},
        "dpb_ms_per_step": {"forward": round(parts["forward"], 4), "backward": round(parts["backward"], 4),
                            "total": round(dpb_ms, 4)},
        "dpb_share": round(dpb_ms / ms, 4),
        "dense_ms_per_step": round(dense_ms, 4) if dense_ms else None,
        "loss": round(loss, 4), "gpu_launches": per_layer * c["layers"] * args.steps, "device_status": status,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default: 1500 for the wide workload, about 2 s; 200 for the "
                         "per-level layouts; 20 for the sweep and the transformer step)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-tokens", type=int, default=2048)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-parity", action="store_true", help="skip the oracle check of sampled rows")
    ap.add_argument("--clock-seconds", type=float, default=2.0,
                    help="a shorter timed region is followed by the same step up to this many seconds, "
                         "so that the clock sampler sees the kernels run")
    ap.add_argument("--e2e-streams", type=int, default=4, help="streams of the host-buffer run")
    ap.add_argument("--no-keep-r", action="store_true", help="backward rebuilds r instead of reading the decode's")
    ap.add_argument("--coset", choices=["wht", "contraction"],
                    help="coset generators g0 ^ {0..15} per level, scored by a WHT or by the contraction")
    ap.add_argument("--e2e-chunks", type=int, default=8,
                    help="chunks of the batch in the host-buffer run (copies overlap kernels across streams)")
    ap.add_argument("--standardise", action="store_true",
                    help="live standardisation tables and the per-step EMA update in the timed step")
    ap.add_argument("--no-dense", action="store_true", help="gpt2small: skip the dense model of the same shape")
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=[WORKLOAD, "tiny", "gpt2", "paper3l", "paper2l", "gpt2small", "sweep"],
                    help="wide (the headline, global selection) or one of the paper's per-level layouts")
    args = ap.parse_args(argv)
    if args.steps is None:
        args.steps = {WORKLOAD: 1500, "paper3l": 200, "paper2l": 200, "tiny": 200, "gpt2": 200}.get(args.workload, 20)
    world, rank, local = dist_env()
    if args.warmup < 3 and args.impl == "ours":
        print("note: at least 3 warm-up steps are used", file=sys.stderr)
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args, world, rank)
    if args.workload == "gpt2small":
        return run_transformer(args, world, rank, local)
    if args.workload == "sweep":
        return run_sweep(args, world, rank, local)
    if args.workload in ("tiny", "gpt2"):
        return run_global_small(args, world, rank, local)
    if args.workload != WORKLOAD:
        return run_per_level(args, world, rank, local)
    return run_ours(args, world, rank, local)


if __name__ == "__main__":
    sys.exit(main())
