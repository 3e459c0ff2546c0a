"""Benchmark of the sparse MLA decode step (VestigeKV hot path) on GB300.

Default workload (the metric's): a Kimi-K2-shaped layer (64 heads, 512 latent + 64 RoPE, bf16 cache), N = 65536
cached rows per sequence, rho = 1/32, r = 64, recent window 256, 64 planted rows per sequence, a batch of 64
independent decode sequences per GPU (weak scaling: every rank owns its own 64 sequences). Metric: decode
query-tokens/s per layer (one query token per sequence per step). ``--config`` selects one of the other evaluation
workloads of datagen.CONFIGS instead (the fp32 tiny layer, the DeepSeek-V2-shaped layers, the log-normal-key layer,
the two-tier layer), with its own selection parameters.

Prints one JSON line (rank 0). `value` times the steps alone (device events on the launching stream); a second
pass of the same steps records the library's stage events for the breakdown and the roofline of the dominant
kernel. `e2e` runs the steps through the same entry point with each step's queries copied in from pinned host
memory and its outputs copied back, on copy streams that overlap the neighbouring steps. On the default workload the
line also carries the sigma selector kernel's throughput over the same cache. `python bench.py --impl reference`
times the CPU oracle on the same workload instead (a bounded sample of sequences per step), on the host cores.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2609_03949_gb300 import datagen  # noqa: E402

DEFAULT_CONFIG = "h64_n64k"
B_PER_GPU = 64                 # sequences per GPU on the default workload
N_DEFAULT = 65536
UNIT = "query-tokens/s"
STAGES = ["qprep", "score", "select", "attn", "trigger", "combine"]


class Workload:
    """The benchmarked workload: sizes, selection parameters and the metric's name."""

    def __init__(self, name: str, B: int | None, N: int | None, rho: float | None, r: int | None, r_sk: int = 0,
                 query_rank: int = 0):
        self.name = name
        self.r_sk, self.query_rank = r_sk, query_rank
        c, p = datagen.CONFIGS[name], datagen.CONFIG_PARAMS[name]
        self.H, self.dtype = c["H"], c["dtype"]
        self.B = B if B is not None else (B_PER_GPU if name == DEFAULT_CONFIG else c["B"])
        self.N = N if N is not None else (N_DEFAULT if name == DEFAULT_CONFIG else c["N"])
        self.rho = rho if rho is not None else p["rho"]
        self.r = r if r is not None else p["r"]
        self.window = p["window"]
        self.trigger = p.get("trigger", 0)
        self.z_eff = p.get("z_eff", 1.0)
        self.n_planted = c["n_planted"]
        self.lognormal = c.get("lognormal_keys", False)
        self.seed = c["seed"]
        n = self.N
        nk = f"{n // 1024}K" if n % 1024 == 0 else str(n)
        rho_s = f"1/{round(1 / self.rho)}" if self.rho < 1 else "1"
        self.metric = f"decode query-tokens/s per layer at N={nk}, rho={rho_s}"
        if name != DEFAULT_CONFIG:
            self.metric += f" ({name})"
        if r_sk:
            self.metric += f" with a rank-{r_sk} content sketch"

    def describe(self, n_gpus: int) -> dict:
        B, N = self.B, self.N
        esz = 2 if self.dtype == "bf16" else 4
        rows = B * N * 576 * esz
        return {"workload": f"sparse MLA decode step: {self.name}, H={self.H}, N={N}, rho={self.rho:g}, r={self.r}, "
                            f"window={self.window}, {self.dtype} cache [512 latent + 64 RoPE]"
                            f"{', two-tier trigger z_eff=%g' % self.z_eff if self.trigger else ''}"
                            f"{', content sketch r_sk=%d' % self.r_sk if self.r_sk else ''}"
                            f"{', content queries of rank %d + 5%% noise' % self.query_rank if self.query_rank else ''}, "
                            f"{self.n_planted} planted rows/seq, B={B} sequences per GPU",
                "heads": self.H, "context": N, "rho": self.rho, "r": self.r, "window": self.window,
                "batch_per_gpu": B, "global_batch": B * n_gpus, "trigger": self.trigger,
                "parallelism": f"independent sequences x{n_gpus} (no collective)",
                "l2": (f"inputs larger than L2: each step streams a {rows / 1e9:.1f} GB cache per GPU (L2 is 129 MB)"
                       if rows >= 4 * 129e6 else
                       f"L2 flushed before every step (512 MB write outside the step's events; the cache is "
                       f"{rows / 1e6:.0f} MB)")}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--config", default=DEFAULT_CONFIG, choices=sorted(datagen.CONFIGS),
                    help="evaluation workload (default: the metric's, H=64, N=65536, rho=1/32, B=64)")
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--context", type=int, default=None, help="cached rows per sequence")
    ap.add_argument("--rho", type=float, default=None)
    ap.add_argument("--r", type=int, default=None, help="score width: 64 or a digest width")
    ap.add_argument("--r-sk", type=int, default=0, help="content sketch rank of the trigger (16, 32, 64; 0 = none)")
    ap.add_argument("--query-rank", type=int, default=0,
                    help="content queries of this rank plus 5%% noise (the sketch basis comes from such prefix queries)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    args.wl = Workload(args.config, args.batch, args.context, args.rho, args.r, args.r_sk, args.query_rank)
    if args.wl.r_sk and not args.wl.trigger:
        ap.error("--r-sk needs a two-tier workload (h128_n64k_two_tier)")
    return args


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_seed(rank: int) -> int:
    """Seed of a rank's own sequences: every rank draws a different, reproducible batch."""
    return 1000 + 7919 * rank


def max_over_ranks(ms: float, pg, device) -> float:
    """The slowest rank's time (the job finishes when its last rank does); a no-op on one process."""
    if pg is None:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def job_throughput(seqs_per_rank: int, world: int, ms_per_step: float) -> float:
    """Whole-job query-tokens/s: every rank's sequences (one query token each) over the slowest rank's step."""
    return seqs_per_rank * world / (ms_per_step * 1e-3)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ------------------------------------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 100 ms while the timed region runs."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.th = threading.Thread(target=self._read, daemon=True)
            self.th.start()
        except (FileNotFoundError, OSError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self, begin: bool):
        if begin:
            self.t0 = time.time()
        else:
            self.t1 = time.time()

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for t, line in self.lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((t, float(parts[1]), float(parts[2]), parts[4:]))
            except ValueError:
                continue
        inside = [r for r in rows if self.t0 is not None and self.t0 - 0.05 <= r[0] <= self.t1 + 0.15]
        use = inside or rows[-3:]
        if not use:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in use for n, v in zip(names, r[3][1:5]) if v.lower() == "active"})
        return {"sm_mhz": float(np.median([r[1] for r in use])), "sm_max_mhz": max(r[2] for r in use),
                "reasons": reasons, "samples": len(use), "in_timed_region": bool(inside)}


def clocks_rejected(clk: dict) -> bool:
    """True when a timed region's clock record rules its number out: a hardware or thermal slowdown was active, or
    the SM clock sat well below its maximum with no reason given (a clock lock left by someone else). sw_power_cap
    alone is kept: it is normal under a long dense load."""
    bad = {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}
    reasons = set(clk.get("reasons") or [])
    if reasons & bad:
        return True
    mhz, top = clk.get("sm_mhz"), clk.get("sm_max_mhz")
    return bool(mhz and top and mhz < 0.8 * top and not (reasons - {"nvidia-smi unavailable", "no samples"}))


# ------------------------------------------------------------------------------------------------ bytes
def union_rows(idx: torch.Tensor, count: torch.Tensor, n: int) -> int:
    """Distinct rows attended per sequence, summed over the batch (ids < 0 or past count are ignored)."""
    B, Hh, cap = idx.shape
    mask = torch.zeros(B, n + 1, dtype=torch.bool, device=idx.device)
    valid = torch.arange(cap, device=idx.device)[None, None, :] < count[..., None]
    ids = torch.where(valid, idx.long(), torch.full_like(idx, n, dtype=torch.long))
    mask.scatter_(1, ids.reshape(B, -1), True)
    return int(mask[:, :n].sum().item())


def kernel_traffic(kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if the kernel's sources are unchanged since."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    d = json.load(open(path)).get(kernel)
    if not d:
        return None
    srcs = [os.path.join(ROOT, f) for f in d["sources"]]
    if not all(os.path.exists(f) for f in srcs):
        return None
    h = hashlib.sha256()
    for f in srcs:
        h.update(open(f, "rb").read())
    if h.hexdigest()[:16] != d["source_sha"]:
        return None
    return float(d["bytes_per_launch"]) * d.get("scale_to_bench", 1.0)


# ------------------------------------------------------------------------------------------------ CPU oracle
N_PREFIX = 512        # prefix queries the sketch basis is computed from


def make_host_workload(w: Workload, B: int, seed: int, device="cpu"):
    return datagen.config_workload(w.name, device=device, B=B, N=w.N, seed=seed, query_rank=w.query_rank)


def oracle_step(hi, digest, w: Workload, basis=None):
    import oracle
    return oracle.decode_step(hi, rho=w.rho, r=w.r, window=w.window, trigger=w.trigger, z_eff=w.z_eff,
                              digest_bf16=digest, sketch_basis=basis)


def oracle_inputs(wl, w: Workload):
    """(host inputs, stored digest, sketch basis) of the oracle's step; the basis from the workload's prefix queries
    (N_PREFIX - 1 of them, so the oracle's Gram route applies)."""
    import oracle
    hi = oracle.HostInputs(wl)
    dig = oracle.build_index(hi, w.r)[1] if w.r < 64 else None
    basis = None
    if w.r_sk:   # the prefix queries depend on the workload's seed alone: one basis per workload
        key = (wl.seed, w.r_sk)
        if key not in _ORACLE_BASIS:
            q = datagen.prefix_queries(wl, N_PREFIX - 1).double().numpy()
            _ORACLE_BASIS[key] = oracle.sketch_basis(q, w.r_sk)[0]
        basis = _ORACLE_BASIS[key]
    return hi, dig, basis


_ORACLE_BASIS = {}


def oracle_baseline(wl_dev, w: Workload, threads: int | None = None, budget_s=12.0, max_seqs=1024):
    """The CPU oracle, as it stands, on a bounded sample of this workload's sequences (host cores, or `threads`)."""
    import oracle
    if threads:
        oracle.set_threads(threads)
    try:
        done, t_total = 0, 0.0
        while done < max_seqs and (t_total < budget_s or done == 0):
            b = done % wl_dev.B
            hi, dig, basis = oracle_inputs(wl_dev.slice_batch([b]), w)
            t0 = time.perf_counter()
            oracle_step(hi, dig, w, basis)
            t_total += time.perf_counter() - t0
            done += 1
            if done == 1 and t_total * max_seqs > 4 * budget_s:
                max_seqs = max(1, int(budget_s / t_total))
        cores = oracle.num_threads()
    finally:
        if threads:
            oracle.set_threads(os.cpu_count() or 1)
    return {"value": done / t_total, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{done} sequence(s) of the bench workload ({w.name}, N={w.N}, H={w.H}) through the fp64 C "
                      f"oracle's whole decode step, {t_total:.1f} s"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import oracle
    w = args.wl
    wl = make_host_workload(w, 2, seed=w.seed)
    inputs = [oracle_inputs(wl.slice_batch([b]), w) for b in range(wl.B)]
    warm = max(3, args.warmup)
    for i in range(warm):
        oracle_step(*inputs[i % 2][:2], w, inputs[i % 2][2])
    t0 = time.perf_counter()
    for i in range(args.steps):
        oracle_step(*inputs[i % 2][:2], w, inputs[i % 2][2])
    dt = time.perf_counter() - t0
    value = args.steps / dt
    line = {"metric": w.metric, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": warm, "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded, bf16 storage)",
            "impl": "reference", "config": w.describe(args.gpus),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                             "sample": f"each step: 1 sequence (N={w.N}, H={w.H}) through the fp64 C oracle"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------------ native
def sigma_throughput(vk, view, B, N, stream, hbm_peak, T=4096, kappa=16, reps=5):
    """The sigma selector kernel over the bench cache (every closed block of T rows): its time and the algorithmic
    bytes (each row's 64 RoPE columns read once, 128 B) against the copy bandwidth."""
    if (N // T) == 0:
        return None
    ws = vk.alloc_bytes(vk.vk_sigma_workspace_bytes(T, kappa))
    sig = torch.empty(B, N, device="cuda")
    for _ in range(2):
        vk.vk_sigma(view, T, kappa, sig, ws)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        vk.vk_sigma(view, T, kappa, sig, ws)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    assert vk.vk_poll_status(ws) == vk.VK_OK
    byts = B * (N // T) * T * 128
    gbs = byts / (ms * 1e-3) / 1e9
    return {"kernel": "k_sigma", "T": T, "kappa": kappa, "blocks": B * (N // T), "ms": ms,
            "algorithmic_bytes": byts, "achieved_gbs": gbs, "frac_of_peak": gbs / hbm_peak,
            "bound": "hbm (two bf16 contractions of 64 x 31 per row: 32 flop/B, below the tensor ridge)"}


def offstep_throughput(vk, view, wl, w, B, N, H, dev, stream, hbm_peak, buf, reps=3):
    """The parts of the method that run off the decode step, on the bench cache, each timed with CUDA events on the
    launching stream (mean of `reps` calls after two warm-up calls), with the algorithmic bytes of its one pass over
    the cache against the copy bandwidth: the PCA digest basis (the RoPE branch's second moment, then a 64 x 64
    eigensolve), the rank-64 content sketch (its basis from the context's prefix queries, then every row's entry) and
    the conformal calibration of z (every (b, h) of the step as a calibration query; its all-rows attention pass
    reads every cached row once)."""
    def timed(fn):
        for _ in range(2):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    def roof(ms, byts):
        gbs = byts / (ms * 1e-3) / 1e9
        return {"algorithmic_bytes": byts, "achieved_gbs": gbs, "frac_of_peak": gbs / hbm_peak}

    out = {}
    rot = torch.empty(64, 64, device=dev)
    eig = torch.empty(64, device=dev)
    pws = vk.alloc_bytes(int(vk.lib().vk_pca_workspace_bytes()))
    ms = timed(lambda: vk.vk_pca_basis(view, rot, eig, pws))
    assert vk.vk_poll_status(pws) == vk.VK_OK
    out["pca"] = {"kernels": "k_pca_moment + k_pca_jacobi", "rows": B * N, "ms": ms, **roof(ms, B * N * 128)}

    q = datagen.prefix_queries(wl, N_PREFIX - 1).to(dev).contiguous()
    basis = torch.empty(64, 512, device=dev)
    sws = vk.vk_sketch_basis(q, 64, basis)
    ms_b = timed(lambda: vk.vk_sketch_basis(q, 64, basis, ws=sws))
    sketch = torch.empty(B, N, 64, dtype=torch.bfloat16, device=dev)
    eta = torch.empty(B, N, device=dev)
    ms_s = timed(lambda: vk.vk_build_sketch(view, 64, basis, sketch, eta))
    out["sketch"] = {"r_sk": 64, "prefix_queries": int(q.shape[0]), "basis_ms": ms_b, "build_kernel": "k_sketch_rows",
                     "build_ms": ms_s, **roof(ms_s, B * N * (1024 + 2 * 64 + 4))}
    del sketch

    params = vk.make_params(w.rho, r=64, window=w.window)
    P = (N + 63) // 64
    pres, pk, pe = (torch.empty(B, P, device=dev) for _ in range(3))
    vk.vk_build_digest(view, params, wl.rot.contiguous(), None, eta, pres, pk, pe)
    index = vk.make_index(None, eta, pres, None, pk, pe)
    buf.run(view, params, index)
    zq = torch.empty(B, H, device=dev)
    z_out = torch.empty(3, device=dev)
    cws = vk.vk_conformal_z(view, params, index, buf.idx, buf.count, zq, z_out)
    ms_c = timed(lambda: vk.vk_conformal_z(view, params, index, buf.idx, buf.count, zq, z_out, ws=cws))
    assert vk.vk_poll_status(cws) == vk.VK_OK
    out["conformal"] = {"queries": B * H, "kernels": "k_attn_tc (all rows, argmax) + k_calib_zq + "
                        "k_conformal_quantile", "ms": ms_c, **roof(ms_c, B * N * 1152)}
    return out


def run_native(args):
    rank, world, local = dist_env()
    if args.gpus != world and world > 1:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE {world}")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    from paper_2609_03949_gb300 import _build, vk
    if rank == 0 or not os.path.exists(vk.LIB_PATH):
        _build.build()
    if pg:
        pg.barrier()
    vk.lib()
    w = args.wl
    B, N, H = w.B, w.N, w.H
    seed = rank_seed(rank) if w.name == DEFAULT_CONFIG else w.seed + 7919 * rank
    wl = make_host_workload(w, B, seed=seed, device=dev)
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    params = vk.make_params(w.rho, r=w.r, window=w.window, trigger=w.trigger, z_eff=w.z_eff, r_sk=w.r_sk)
    # the per-cache index (built once, off the step): digest for r < 64, norms for the trigger
    index = None
    if w.r < 64 or w.trigger:
        P = (N + 63) // 64
        dig = torch.empty(B, N, w.r, dtype=torch.bfloat16, device=dev) if w.r < 64 else None
        rot = wl.rot.contiguous()
        eta = torch.empty(B, N, device=dev)
        pres, pk, pe = (torch.empty(B, P, device=dev) for _ in range(3))
        vk.vk_build_digest(view, params, rot, dig, eta, pres, pk, pe)
        sketch = basis = None
        if w.r_sk:
            # V from the context's prefix queries, then every row's sketch entry (eta becomes the sketch residual)
            q = datagen.prefix_queries(wl, N_PREFIX - 1).to(dev).contiguous()
            basis = torch.empty(w.r_sk, 512, device=dev)
            vk.vk_sketch_basis(q, w.r_sk, basis)
            sketch = torch.empty(B, N, w.r_sk, dtype=torch.bfloat16, device=dev)
            vk.vk_build_sketch(view, w.r_sk, basis, sketch, eta)
        index = vk.make_index(dig, eta, pres, rot if w.r < 64 else None, pk, pe, sketch, basis)
    buf = vk.DecodeBuffers(view, params, device=dev)
    stream = torch.cuda.current_stream(dev)

    # ---- device-timed region: inputs resident in HBM, per-stage CUDA events on the launching stream
    for _ in range(max(3, args.warmup)):
        buf.run(view, params, index)
    torch.cuda.synchronize()
    assert vk.vk_poll_status(buf.ws) == vk.VK_OK
    step_events = [[torch.cuda.Event(enable_timing=True) for _ in range(7)] for _ in range(args.steps)]
    step_brackets = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    for evs in step_events + step_brackets:   # create the underlying cudaEvent_t handles outside the timed region
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize()
    esz = 2 if w.dtype == "bf16" else 4
    # a cache that L2 could hold is evicted between steps by a 512 MB write outside the steps' events
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev) if B * N * 576 * esz < 4 * 129e6 else None
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)

    def headline_pass():
        # the steps alone (no stage events), bracketed by events on the launching stream; with an L2 flush between
        # steps, each step is bracketed by its own pair so that the flushes stay outside
        clocks = ClockSampler(local)
        clocks.start()
        time.sleep(0.3)
        if pg:
            pg.barrier()
        torch.cuda.synchronize()
        launches0 = vk.vk_profile_launches()
        clocks.mark(True)
        t_start.record(stream)
        for sb, se in step_brackets:
            if flush is not None:
                flush.fill_(1)
                sb.record(stream)
            buf.run(view, params, index)
            if flush is not None:
                se.record(stream)
        t_end.record(stream)
        torch.cuda.synchronize()
        clocks.mark(False)
        n_launch = vk.vk_profile_launches() - launches0
        ms = t_start.elapsed_time(t_end)
        if flush is not None:
            ms = sum(sb.elapsed_time(se) for sb, se in step_brackets)
        return max_over_ranks(ms, pg, dev), n_launch, clocks.stop()

    # pass 1, the headline; taken once more if any rank's clock record rules it out
    elapsed_ms, launches, clk = headline_pass()
    if max_over_ranks(1.0 if clocks_rejected(clk) else 0.0, pg, dev) > 0:
        first = clk
        elapsed_ms, launches, clk = headline_pass()
        clk = dict(clk, remeasured_after=first)
    ms_step = elapsed_ms / args.steps
    assert vk.vk_poll_status(buf.ws) == vk.VK_OK
    # pass 2, the breakdown: the same steps again, each recording its stage boundaries into its own events
    stage_ms = np.zeros(6)
    total_ms_events = 0.0
    for evs in step_events:
        if flush is not None:
            flush.fill_(1)
        vk.vk_profile_set_events(evs)
        buf.run(view, params, index)
    torch.cuda.synchronize()
    vk.vk_profile_set_events([])
    for evs in step_events:
        for i in range(6):
            stage_ms[i] += evs[i].elapsed_time(evs[i + 1])
        total_ms_events += evs[0].elapsed_time(evs[6])
    assert vk.vk_poll_status(buf.ws) == vk.VK_OK
    dev_ms_step = total_ms_events / args.steps
    stage_ms /= args.steps

    # ---- algorithmic bytes (distinct rows gathered per sequence, summed; the trigger's scan and new fired rows)
    from paper_2609_03949_gb300.bytes_model import row_bytes, score_bytes_per_row, step_bytes
    k = vk.vk_keep_count(N, w.rho, w.window, 0)
    nS = k + w.window
    U1 = union_rows(buf.idx[..., :nS], torch.minimum(buf.count, torch.tensor(nS, device=dev)), N)
    U = union_rows(buf.idx, buf.count, N) if w.trigger else U1
    step_b = step_bytes(N, B, w.r, w.dtype, U1, bool(w.trigger), U - U1, w.r_sk)
    hbm_peak, peak_kind = peaks()
    sb = score_bytes_per_row(w.r, w.dtype)
    stage_bytes = {"score": B * N * sb, "attn": U1 * row_bytes(w.dtype),
                   "trigger": B * N * (sb + 4 + 2 * w.r_sk) + (U - U1) * row_bytes(w.dtype)}
    cands = ["score", "attn"] + (["trigger"] if w.trigger else [])
    dom = max(cands, key=lambda st: stage_ms[STAGES.index(st)])
    dom_ms = stage_ms[STAGES.index(dom)]
    achieved = stage_bytes[dom] / (dom_ms * 1e-3) / 1e9
    roof = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
            "frac": achieved / hbm_peak, "peak_kind": f"{peak_kind} copy bandwidth",
            "traffic": kernel_traffic(dom) if (w.name, B, N) == (DEFAULT_CONFIG, B_PER_GPU, N_DEFAULT) else None,
            "algorithmic_bytes_per_launch": stage_bytes[dom], "ms_per_launch": dom_ms}

    # ---- end to end through the public C entry point with host buffers (pinned). Every step copies its queries
    # in from pinned host memory and its outputs back; the copies run on their own streams and overlap the
    # neighbouring steps' kernels (two query/output buffer sets, ordered by events), as a serving loop would.
    qlh = wl.q_latent.cpu().pin_memory()
    qrh = wl.q_rope.cpu().pin_memory()
    qls = [torch.empty_like(wl.q_latent) for _ in range(2)]
    qrs = [torch.empty_like(wl.q_rope) for _ in range(2)]
    views = [vk.make_view(wl.cache, qls[k], qrs[k]) for k in range(2)]
    bufs = [buf, vk.DecodeBuffers(views[1], params, device=dev)]
    outh = [torch.empty_like(buf.out, device="cpu").pin_memory() for _ in range(2)]
    lseh = [torch.empty_like(buf.lse, device="cpu").pin_memory() for _ in range(2)]
    h2d = qlh.numel() * qlh.element_size() + qrh.numel() * qrh.element_size()
    d2h = outh[0].numel() * outh[0].element_size() + lseh[0].numel() * lseh[0].element_size()
    s_in = torch.cuda.Stream(dev)
    s_out = torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(2)]      # queries of buffer k landed
    ev_comp = [torch.cuda.Event() for _ in range(2)]    # step on buffer k done
    ev_out = [torch.cuda.Event() for _ in range(2)]     # outputs of buffer k copied out

    def e2e_steps(n):
        for i in range(n):
            k = i & 1
            if i >= 2:
                s_in.wait_event(ev_comp[k])              # step i - 2 has read these query buffers
            with torch.cuda.stream(s_in):
                qls[k].copy_(qlh, non_blocking=True)
                qrs[k].copy_(qrh, non_blocking=True)
                ev_in[k].record(s_in)
            stream.wait_event(ev_in[k])
            if i >= 2:
                stream.wait_event(ev_out[k])             # step i - 2's outputs are out of these buffers
            bufs[k].run(views[k], params, index)
            ev_comp[k].record(stream)
            s_out.wait_event(ev_comp[k])
            with torch.cuda.stream(s_out):
                outh[k].copy_(bufs[k].out, non_blocking=True)
                lseh[k].copy_(bufs[k].lse, non_blocking=True)
                ev_out[k].record(s_out)
        for k in range(min(n, 2)):
            stream.wait_event(ev_out[k])

    e2e_steps(3)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_in.wait_event(e0)
    s_out.wait_event(e0)
    e2e_steps(args.steps)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    e2e_ms = max_over_ranks(e2e_ms, pg, dev)
    assert all(torch.isfinite(t).all() for t in lseh)
    assert vk.vk_poll_status(bufs[1].ws) == vk.VK_OK

    sigma = offstep = None
    if w.name == DEFAULT_CONFIG and w.dtype == "bf16":
        sigma = sigma_throughput(vk, view, B, N, stream, hbm_peak)
        offstep = offstep_throughput(vk, view, wl, w, B, N, H, dev, stream, hbm_peak, buf)

    cpu = cpu1 = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = oracle_baseline(wl, w)
        cpu1 = oracle_baseline(wl, w, threads=1, budget_s=6.0)

    line = {
        "metric": w.metric, "value": job_throughput(B, world, ms_step), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
        "data": f"synthetic (seeded Gaussian MLA cache, {w.dtype})", "config": w.describe(world),
        "roofline": roof, "cpu_baseline": cpu, "cpu_baseline_single_thread": cpu1,
        "e2e": {"value": job_throughput(B, world, e2e_ms / args.steps), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches), "clocks": clk,
        "step": {"device_ms_per_step": dev_ms_step, "algorithmic_bytes": step_b,
                 "hbm_gbs": step_b / (ms_step * 1e-3) / 1e9, "frac_of_peak": step_b / (ms_step * 1e-3) / 1e9 / hbm_peak,
                 "union_rows_per_seq": U1 / B, "union_frac": U1 / (B * N),
                 "fired_new_rows_per_seq": (U - U1) / B,
                 "stage_ms": {st: float(stage_ms[i]) for i, st in enumerate(STAGES)}},
        "sigma": sigma,
        "offstep": offstep,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
