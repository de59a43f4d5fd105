#!/usr/bin/env python
"""Benchmark: one synthetic Llama-shaped linear layer through the KronQ per-layer path
(factors -> BiIP rescale + RHT -> damped inverse Cholesky -> OBS sweep) per step.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config down_70b] [--impl ours|reference]

Prints one JSON line. `value` is milliseconds per linear layer for the whole job (lower is
better). Under torchrun each rank quantizes its own layer (the path has no cross-layer
exchange: weak scaling, no collective on the data path); the timed region is bracketed by
a barrier and a device synchronize on every rank and the slowest rank's time is used.
`--impl reference` times the CPU oracle (float64 numpy + the fp32-ordered C sweep) on a
bounded sample of the same workload and extrapolates to the same metric.
"""
from __future__ import annotations

import argparse
import datetime
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import kqsynth  # noqa: E402
import numpy as np  # noqa: E402

METRIC = "ms per linear layer (factors+rotate+chol+OBS sweep)"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default: 100 for a layer or decode, 10 for a block, 3 for the oracle arm)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default="down_70b", choices=sorted(kqsynth.CONFIGS),
                    help="layer workload (default: the largest, Llama-3-70B down_proj 8192 x 28672)")
    ap.add_argument("--secondary", default="q_proj_8b",
                    help="a second layer shape measured in the same run and reported under 'secondary' "
                         "('' for none)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="launch kernels directly instead of replaying a CUDA graph")
    ap.add_argument("--x-chunk-tokens", type=int, default=0,
                    help="token chunk of the H_X accumulation (0: one call)")
    ap.add_argument("--g-chunk-tokens", type=int, default=0,
                    help="token chunk of the H_G accumulation with device-resident inputs (0: one call)")
    ap.add_argument("--e2e-x-chunk-tokens", type=int, default=None,
                    help="token chunk of the H_X accumulation on the host path, each chunk started as soon as "
                         "its copy has landed (default: 32768 when X is larger than 4 GiB, else one call)")
    ap.add_argument("--e2e-g-chunk-tokens", type=int, default=32768,
                    help="token chunk of the H_G accumulation on the host path, where each chunk starts "
                         "as soon as its copy has landed (0: one call)")
    ap.add_argument("--trailing", default="3xtf32", choices=["fp32", "3xtf32"],
                    help="sweep trailing update: fp32-ordered SIMT (bit-exact) or 3xTF32 tensor cores")
    ap.add_argument("--block", default=None, choices=sorted(kqsynth.BLOCKS),
                    help="a whole transformer block (seven sublayers, shared H_X, W2/W3 allocation) "
                         "instead of one layer")
    ap.add_argument("--lanes", type=int, default=2, help="sublayers quantized concurrently in --block mode")
    ap.add_argument("--infer", type=int, default=None, metavar="BITS",
                    help="decode with quantized layers instead: one token through every linear sublayer of "
                         "--infer-blocks Llama-3-8B blocks (kq_infer, online BiIP revert)")
    ap.add_argument("--infer-blocks", type=int, default=32)
    ap.add_argument("--validate", action="store_true",
                    help="Prop. 2 checks on the --config layer: output-side exponent sweep of the rescale, "
                         "rho, CV of column/row norms (not a timing run)")
    ap.add_argument("--infer-tokens", type=int, default=1)
    ap.add_argument("--drift-chunk-tokens", type=int, default=0,
                    help="token chunk of the drift statistic's launches (0: one launch)")
    ap.add_argument("--tokens", type=int, default=0,
                    help="override the workload's token count (small cases for profiling captures)")
    ap.add_argument("--drift", type=float, default=None, metavar="ALPHA",
                    help="with the GPTAQ drift correction of scaling ALPHA (full-precision input X~ = "
                         "X + 0.1 sigma z); default: GPTQ mode")
    args = ap.parse_args()
    if args.steps is None:
        # a timed region of several seconds, so that the clock record has samples inside it
        # (a down_70b layer takes ~0.4 s, a q_proj layer ~6 ms)
        big = kqsynth.CONFIGS[args.config].d_in * kqsynth.CONFIGS[args.config].d_out > (64 << 20)
        args.steps = 3 if args.impl == "reference" else 10 if args.block else 20 if big else 100
    return args


def metric_of(alpha) -> str:
    return METRIC if alpha is None else "ms per linear layer (factors+drift+rotate+chol+P+OBS sweep)"


def workload_name(cfg) -> str:
    return (f"{cfg.name}: W {cfg.d_out}x{cfg.d_in}, T={cfg.T} tokens, {cfg.bits}-bit "
            f"{'per-row' if cfg.group == 0 else 'group ' + str(cfg.group)}, block {cfg.block}, "
            f"damp {cfg.damp}")


def config_dict(cfg, x_chunk: int = 0, g_chunk: int = 0, trailing: str = "3xtf32", alpha=None) -> dict:
    d = {"workload": workload_name(cfg), "d_out": cfg.d_out, "d_in": cfg.d_in, "T": cfg.T,
         "bits": cfg.bits, "group": cfg.group, "block": cfg.block, "damp": cfg.damp,
         "factor_chunk_tokens": {"X": x_chunk, "G": g_chunk}, "sweep_trailing_update": trailing,
         "l2": "inputs larger than L2 (X and G are T x d bf16, >= 1 GiB each); no flush"}
    if alpha is not None:
        d["workload"] += f" + GPTAQ drift correction (alpha {alpha}, X~ = X + 0.1 sigma z)"
        d["drift_alpha"] = alpha
    return d


def algorithmic_flops(cfg, drift: bool = False) -> dict:
    fl = {"factor_x": cfg.T * cfg.d_in * (cfg.d_in + 1),
          "factor_g": cfg.T * cfg.d_out * (cfg.d_out + 1),
          "chol": 2 * cfg.d_in ** 3 / 3,
          "sweep": cfg.d_out * cfg.d_in * max(cfg.d_in - cfg.block, 0) * (2 if drift else 1)}
    if drift:
        fl["drift"] = 2 * cfg.T * cfg.d_in ** 2       # (X~ - X)^T X
        fl["p"] = 2 * cfg.d_in ** 3 / 3               # two triangular products
    return fl


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def syrk_traffic(cfg, launch_tokens: int):
    """DRAM bytes per SYRK launch from a committed ncu capture of a launch of the same
    shape (d, tokens per launch), taken on the current kernel source; else None."""
    src = os.path.join(ROOT, "paper_2607_07964_gb300", "csrc", "syrk.cu")
    rec = os.path.join(ROOT, "profiles", "syrk_traffic.json")
    try:
        with open(rec) as f:
            r = json.load(f)
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if r.get("syrk_cu_sha256_16") != h or r.get("d") != cfg.d_in or r.get("T") != launch_tokens:
            return None
        return float(r["dram_bytes_per_launch"])
    except (OSError, ValueError, KeyError):
        return None


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap,pci.bus_id")

    def __init__(self, bus_id: str | None):
        self.bus_id = (bus_id or "").lower()
        self.proc = None
        self.path = None

    def start(self):
        """Start sampling and return once the first sample is written (bounded by 5 s), so
        that the samples taken after this call cover the timed region that follows."""
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
            return
        t_end = time.time() + 5.0
        while time.time() < t_end and self.proc.poll() is None and os.path.getsize(self.path) == 0:
            time.sleep(0.01)
        self.t_begin = datetime.datetime.now()

    def stop(self) -> dict | None:
        """Clock record of the region between start() and this call: the samples stamped
        inside it, or, for a region shorter than the sampling period, the first sample
        stamped after it began."""
        if self.proc is None:
            return None
        t_stop = datetime.datetime.now()
        time.sleep(0.25)   # lets a region shorter than the period receive its sample
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        rows = []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            if self.bus_id and not f[8].lower().endswith(self.bus_id[-12:]):
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f")
                rows.append((ts, float(f[1]), float(f[2]), [n for k, n in enumerate(names)
                                                            if f[4 + k].lower() == "active"]))
            except ValueError:
                continue
        os.unlink(self.path)
        inside = [r for r in rows if self.t_begin <= r[0] <= t_stop]
        if not inside:
            inside = [r for r in rows if r[0] >= self.t_begin][:1]
        if not inside:
            return None
        return {"sm_mhz": statistics.median(r[1] for r in inside), "sm_max_mhz": max(r[2] for r in inside),
                "samples": len(inside), "reasons": sorted({n for r in inside for n in r[3]}),
                "region_ms": round((t_stop - self.t_begin).total_seconds() * 1e3, 1)}


# ---------------------------------------------------------------- CPU oracle timing
# Bounded samples of the oracle, per stage: the factors on T_s and 2 T_s of the T tokens at
# full width (a line in the tokens), the BiIP dense products and the textbook inverse
# Cholesky on the layer shrunk by f in both dimensions (cubic in the size), the fp32-ordered
# sweep on rows_s rows of that shrunk layer (proportional to rows x d_in^2). f = 1 runs
# BiIP and the Cholesky at full size.
ORACLE_SAMPLES = {
    "large": dict(T_s=2048, f=4, rows_s=64),
    "medium": dict(T_s=1024, f=8, rows_s=64),
    "small": dict(T_s=512, f=16, rows_s=32),
}


def _shrink(cfg, f: int) -> int:
    """The largest of f, f/2, ... (down to 1) that leaves both dimensions >= 256 and keeps
    the Hadamard sizes (2^k or 28 * 2^k) whole."""
    while f > 1 and (min(cfg.d_in, cfg.d_out) // f < 256 or cfg.d_in % f or cfg.d_out % f):
        f //= 2
    return max(f, 1)


def two_point_tokens(t1: float, t2: float, T_s: int, T: int) -> float:
    """Time for T tokens from times t1, t2 on T_s and 2 T_s tokens: the line through both,
    or t2 scaled by T / (2 T_s) when t2 <= t1 (no usable slope)."""
    slope = (t2 - t1) / T_s
    return t2 + (T - 2 * T_s) * slope if slope > 0 else t2 * T / (2 * T_s)


def _oracle_stages(cfg, T_s: int, f: int, rows_s: int, alpha=None) -> dict:
    """One timed pass of every stage on its sample, each extrapolated to the full layer (ms)."""
    from oracle import kronq_oracle as ref
    import oracle

    T_s = min(cfg.T, T_s)
    f = _shrink(cfg, f)
    sub = cfg.replace(d_out=cfg.d_out // f, d_in=cfg.d_in // f, T=T_s)
    rows_s = min(sub.d_out, rows_s)
    L = {"X": kqsynth.activations(cfg, 2 * T_s), "G": kqsynth.gradients(cfg, 2 * T_s)}
    Ls = kqsynth.layer(sub) if f > 1 else dict(L, W=kqsynth.weights(cfg), **dict(zip(("sign_u", "sign_v"),
                                                                                   kqsynth.signs(cfg))))
    drift = alpha is not None
    per = {}
    # the factors on T_s and on 2 T_s tokens, after an untimed call that starts the library's
    # threads: a d x d result costs the same at any T (its allocation and write), so the
    # full layer is the two-point line through both times. Where the second time is not the
    # larger (the fixed part varied between the calls by more than the tokens' part), the
    # line has no usable slope and the larger sample is scaled in proportion to the tokens.
    ref.accum_factor(L["G"][:min(64, T_s)])
    tf = []
    for Tk in (T_s, 2 * T_s):
        t0 = time.perf_counter()
        ref.accum_factor(L["X"][:Tk])
        ref.accum_factor(L["G"][:Tk])
        tf.append(time.perf_counter() - t0)
    per["factors"] = two_point_tokens(tf[0], tf[1], T_s, cfg.T)
    Ds = None
    if drift:
        Xt = kqsynth.fp_activations(cfg, L["X"])
        t1 = time.perf_counter()
        ref.drift_factor(Xt, L["X"])
        per["drift"] = (time.perf_counter() - t1) * cfg.T / T_s
        Ds = ref.drift_factor(kqsynth.fp_activations(sub, Ls["X"]), Ls["X"])
    HXs, HGs = ref.accum_factor(Ls["X"]), ref.accum_factor(Ls["G"])
    t1 = time.perf_counter()
    b = ref.biip(Ls["W"], HXs, HGs, Ls["sign_u"], Ls["sign_v"], Ds)
    t2 = time.perf_counter()
    per["biip"] = (t2 - t1) * f ** 3
    R = ref.inverse_cholesky_upper(ref.damp(b["HX"], cfg.damp))
    t3 = time.perf_counter()
    per["chol"] = (t3 - t2) * f ** 3
    Pt = None
    if drift:
        P = ref.gptaq_p(b["D"], R.T, alpha)
        per["p"] = (time.perf_counter() - t3) * f ** 3
        Pt = P.T.astype("float32")
    Wp = np.ascontiguousarray(b["W"][:rows_s]).astype("float32")
    Lt = R.T.astype("float32")
    t4 = time.perf_counter()
    oracle.obs_sweep_fp32(Wp, Lt, cfg.bits, cfg.group, cfg.block, Pt=Pt)
    per["sweep"] = (time.perf_counter() - t4) * (cfg.d_out / rows_s) * f ** 2
    return {"stages_ms": {k: 1e3 * v for k, v in per.items()}, "T_s": T_s, "f": f, "rows_s": rows_s}


def oracle_sample_ms(cfg, preset: str = "large", alpha=None, check: bool = True) -> dict:
    """The oracle's time for the layer from the `preset` sample, and (check) the same
    estimate from a sample half as large (half the tokens, twice the shrink, half the
    rows), stage by stage, with their ratio: the cost models hold where the two agree."""
    kw = ORACLE_SAMPLES[preset]
    main = _oracle_stages(cfg, kw["T_s"], kw["f"], kw["rows_s"], alpha)
    per = main["stages_ms"]
    out = {"value": sum(per.values()), "unit": "ms", "cores": os.cpu_count(), "kind": "oracle",
           "stages_ms": per, "preset": preset,
           "sample": (f"factors on {main['T_s']} and {2 * main['T_s']} of {cfg.T} tokens at full width (two-point "
                      f"line to {cfg.T}); "
                      f"BiIP dense products and textbook inverse Cholesky on the {cfg.d_out // main['f']}x"
                      f"{cfg.d_in // main['f']} layer (x{main['f']}^3); fp32-ordered sweep on {main['rows_s']} rows "
                      f"of it (x{main['f']}^2*{cfg.d_out / main['rows_s']:g})"
                      + ("; drift statistic on the factors' tokens, P on the shrunk layer" if alpha is not None
                         else ""))}
    if check:
        # half the tokens and twice the shrink; the same rows (the fp32 sweep runs rows in
        # parallel, so fewer rows than a few per core would change the cost per row)
        half = _oracle_stages(cfg, max(1, kw["T_s"] // 2), 2 * kw["f"], kw["rows_s"], alpha)
        out["check"] = {"sample": f"T_s {half['T_s']}, shrink {half['f']}, {half['rows_s']} rows",
                        "stages_ms": half["stages_ms"],
                        "ratio": {k: per[k] / half["stages_ms"][k] for k in per if half["stages_ms"][k] > 0}}
    return out


# --------------------------------------------------------------------- distributed
def dist_setup(backend: str):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)
    return ws, rank, local


def max_over_ranks(v: float, ws: int, device: str = "cpu") -> float:
    """The slowest rank's value (the job's time); v itself when there is one rank."""
    if ws <= 1:
        return v
    import torch
    t = torch.tensor([v], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def reference_preset(steps: int, warmup: int) -> str:
    """The oracle sample per step of the reference arm: the same sample as our line's
    cpu_baseline ("large") when the run has few steps, smaller ones when many steps would
    otherwise run past a few minutes."""
    n = steps + warmup
    return "large" if n <= 6 else "medium" if n <= 16 else "small"


def run_reference(args):
    ws, rank, _ = dist_setup("gloo")
    cfg = kqsynth.CONFIGS[args.config]
    if args.tokens > 0:
        cfg = cfg.replace(T=args.tokens)
    if rank != 0:
        return
    preset = reference_preset(args.steps, args.warmup)
    for _ in range(args.warmup):
        oracle_sample_ms(cfg, preset, args.drift, check=False)
    vals, first = [], None
    t0 = time.perf_counter()
    for k in range(args.steps):
        r = oracle_sample_ms(cfg, preset, args.drift, check=(k == 0))
        first = first or r
        vals.append(r["value"])
    wall = time.perf_counter() - t0
    v = statistics.mean(vals)
    cpu = dict(first, value=v, steps_ms=vals)
    out = {"impl": "reference", "metric": metric_of(args.drift), "value": v, "unit": "ms", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": v, "higher_is_better": False,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": config_dict(cfg, args.x_chunk_tokens, args.g_chunk_tokens, args.trailing, args.drift),
           "cpu_baseline": cpu,
           "e2e": {"value": v, "unit": "ms", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
           "timing": "each step times the oracle on a bounded sample of the layer and extrapolates every "
                     "stage to the full layer by its cost model (see cpu_baseline.sample and .check)",
           "wall_s": wall}
    print(json.dumps(out), flush=True)


def tf32_peak(peaks: dict) -> tuple[float, str]:
    """Dense tf32 tensor peak: the measured bf16 burst times the nominal tf32 : bf16 ratio
    (1.1 : 2.25 PFLOP/s dense)."""
    bf16 = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    return bf16 * 1.1 / 2.25, "measured bf16 dense burst x 1.1/2.25 (nominal tf32 : bf16)"


def rotation_bytes(cfg) -> dict:
    """Bytes of the rotation stage: algorithmic (each two-sided transform of an fp32 matrix
    read and written once: H_X' 8 d_in^2, H_G' 8 d_out^2, W' 8 d_out d_in) and moved by this
    implementation (H_X and H_G: row pass, transpose, row pass; W: copy into the work
    buffer, row pass, column pass)."""
    hx, hg, w = 4 * cfg.d_in ** 2, 4 * cfg.d_out ** 2, 4 * cfg.d_out * cfg.d_in
    return {"algorithmic": 2 * (hx + hg + w), "moved": 2 * 3 * (hx + hg) + 2 * 3 * w}


def fractions(cfg, stage_ms: dict, peaks: dict, peak_src: str) -> dict:
    """Per-stage throughput against the roofline that bounds it: the SYRKs against the bf16
    tensor peak, the Cholesky and the sweep's trailing update against the tf32 peak
    (algorithmic flops, and executed: the 3xTF32 split runs three tf32 products per
    multiply-add), the rotations against HBM bandwidth."""
    bf16 = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    tf32, tf32_src = tf32_peak(peaks)
    fl = algorithmic_flops(cfg)
    out = {"peaks": {"bf16_tflops": bf16, "tf32_tflops": tf32, "hbm_gbs": hbm,
                     "source": f"{peak_src}; tf32 = {tf32_src}"}}
    bf16_s = float(peaks.get("bf16_tflops_sustained", bf16))
    out["peaks"]["bf16_tflops_sustained"] = bf16_s
    for k in ("factor_x", "factor_g"):
        t = fl[k] / stage_ms[k] / 1e9
        out[k] = {"tflops": t, "frac_bf16": t / bf16, "frac_bf16_sustained": t / bf16_s}
    for k, name in (("chol", "chol"), ("sweep", "sweep_trailing")):
        t = fl[k] / stage_ms[k] / 1e9
        out[name] = {"tflops_algorithmic": t, "frac_tf32_algorithmic": t / tf32,
                     "tflops_executed_3xtf32": 3 * t, "frac_tf32_executed": 3 * t / tf32}
    rb = rotation_bytes(cfg)
    ga, gm = rb["algorithmic"] / stage_ms["rotate"] / 1e6, rb["moved"] / stage_ms["rotate"] / 1e6
    out["rotate"] = {"gbs_algorithmic": ga, "frac_hbm_algorithmic": ga / hbm, "gbs_moved": gm,
                     "frac_hbm_moved": gm / hbm, "bytes_algorithmic": rb["algorithmic"], "bytes_moved": rb["moved"]}
    return out


def h2d_link_probe(dev, nbytes: int = 1 << 31, reps: int = 3) -> dict:
    """Host-to-device bandwidth from pinned memory: the same bytes copied on one stream, and
    split evenly over 2 and 4 streams running at once (best of `reps`, CUDA events)."""
    import torch

    host = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    devb = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    out = {}
    for ns in (1, 2, 4):
        streams = [torch.cuda.Stream(device=dev) for _ in range(ns)]
        per = nbytes // ns
        best = float("inf")
        for _ in range(reps):
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            cur = torch.cuda.current_stream()
            e0.record(cur)
            for k, st in enumerate(streams):
                st.wait_event(e0)
                with torch.cuda.stream(st):
                    devb[k * per:(k + 1) * per].copy_(host[k * per:(k + 1) * per], non_blocking=True)
            for st in streams:
                cur.wait_stream(st)
            e1.record(cur)
            torch.cuda.synchronize()
            best = min(best, e0.elapsed_time(e1))
        out[f"{ns}_streams"] = nbytes / best / 1e6
    del host, devb
    return {"bytes": nbytes, "gbs": out}


def measure_layer(cfg, args, dev, ws, steps, stream, barrier, sample_clocks: bool = True):
    """Warm-up, then `steps` timed graph replays (or direct runs) of one layer, then a
    serialized pass with per-stage events. Returns the timings and the pipeline."""
    import torch

    from paper_2607_07964_gb300 import kronq as kq
    from paper_2607_07964_gb300.pipeline import LayerPipeline

    inp = kqsynth.device_layer(cfg, device=dev)
    drift = args.drift is not None
    Xt = kqsynth.device_fp_activations(cfg, inp["X"]) if drift else None
    p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, device=dev,
                      x_chunk_tokens=args.x_chunk_tokens, g_chunk_tokens=args.g_chunk_tokens,
                      trailing=args.trailing, alpha=args.drift, drift_chunk_tokens=args.drift_chunk_tokens)
    run_args = (inp["X"], inp["G"], inp["W"], inp["sign_u"], inp["sign_v"])
    for _ in range(args.warmup):
        p.run(*run_args, stream=stream, Xt=Xt)
    p.check(stream)
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    props = torch.cuda.get_device_properties(dev)
    sampler = ClockSampler(getattr(props, "pci_bus_id", None))
    barrier()
    torch.cuda.synchronize()
    graph = None
    per_step = 0
    if not args.no_graph:
        graph, per_step = p.capture(*run_args, Xt=Xt)
        for _ in range(2):
            graph.replay()
        torch.cuda.synchronize()
        barrier()
    if sample_clocks:
        sampler.start()
    n0 = kq.launch_count()
    t_start.record(stream)
    for _ in range(steps):
        if graph is not None:
            graph.replay()
        else:
            p.run(*run_args, stream=stream, Xt=Xt)
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = per_step * steps if graph is not None else kq.launch_count() - n0
    clocks = sampler.stop() if sample_clocks else None
    p.check(stream)
    total_ms = max_over_ranks(t_start.elapsed_time(t_end), ws, dev)
    del graph
    # Per-stage times come from a second, serialized pass (each stage alone on the stream,
    # bracketed by events); the headline value above overlaps stages.
    n_ser = max(1, min(steps, 10))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(p.stages) + 1)] for _ in range(n_ser)]
    torch.cuda.synchronize()
    for k in range(n_ser):
        p.run(*run_args, stream=stream, events=evs[k], Xt=Xt)
    torch.cuda.synchronize()
    p.check(stream)
    stage_ms = {name: statistics.mean(evs[k][i].elapsed_time(evs[k][i + 1]) for k in range(n_ser))
                for i, name in enumerate(p.stages)}
    return {"total_ms": total_ms, "stage_ms": stage_ms, "launches": launches, "clocks": clocks,
            "graph": not args.no_graph, "pipeline": p, "inputs": inp, "Xt": Xt}


def run_ours(args):
    import torch

    from paper_2607_07964_gb300 import build as kbuild
    ws, rank, local = dist_setup("nccl")
    kbuild.build()
    from paper_2607_07964_gb300.pipeline import LayerPipeline

    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    cfg = kqsynth.CONFIGS[args.config].replace(seed=rank)
    if args.tokens > 0:
        cfg = cfg.replace(T=args.tokens)
    drift = args.drift is not None
    stream = torch.cuda.current_stream()

    def barrier():
        if ws > 1:
            torch.distributed.barrier()

    steps = args.steps
    m = measure_layer(cfg, args, dev, ws, steps, stream, barrier)
    p, inp, Xt = m["pipeline"], m["inputs"], m["Xt"]
    stage_ms, total_ms, launches, clocks = m["stage_ms"], m["total_ms"], m["launches"], m["clocks"]
    used_graph = m["graph"]
    fl = algorithmic_flops(cfg, drift)
    tflops = {"factor_x": fl["factor_x"] / stage_ms["factor_x"] / 1e9,
              "factor_g": fl["factor_g"] / stage_ms["factor_g"] / 1e9,
              "chol": fl["chol"] / stage_ms["chol"] / 1e9,
              "sweep_trailing": fl["sweep"] / stage_ms["sweep"] / 1e9}
    if drift:
        tflops["drift"] = fl["drift"] / stage_ms["drift"] / 1e9
        tflops["p"] = fl["p"] / stage_ms["p"] / 1e9
    peaks, peak_src = measured_peaks()
    burst = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    sustained = float(peaks.get("bf16_tflops_sustained", burst))
    # factor_x is one SYRK launch per token chunk: flops per launch / mean launch time.
    n_launch = len(p._chunks("X", cfg.T))
    achieved = tflops["factor_x"]
    traffic = syrk_traffic(cfg, cfg.T // n_launch)
    # A launch of tens of milliseconds inside back-to-back layer steps runs under the power
    # cap: its peak is the sustained figure; a short launch is compared with the burst one.
    long_launch = stage_ms["factor_x"] / n_launch >= 10.0
    peak = sustained if long_launch else burst
    roofline = {"kernel": "syrk_tc_kernel (H_X = X^T X)", "bound": "tensor", "achieved": achieved,
                "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
                "peak_source": (f"{peak_src} bf16 dense sustained (of measured: the launch lasts "
                                f"{stage_ms['factor_x'] / n_launch:.0f} ms inside back-to-back layer steps)"
                                if long_launch else f"{peak_src} bf16 dense burst (of measured)"),
                "frac_of_burst": achieved / burst, "frac_of_sustained": achieved / sustained,
                "algorithmic_flops_per_launch": fl["factor_x"] / n_launch, "launches_per_factor": n_launch,
                "timing": "CUDA events around the H_X stage of the serialized pass (one launch, on its stream)"}
    if drift:
        # the drift stage (one split pass + one drift_tc_kernel launch with K = 2 T): algorithmic
        # flops of (X~ - X)^T X over the stage time; the split pair executes twice as many
        a = tflops["drift"]
        roofline = {"kernel": "drift stage (drift_split_kernel + drift_tc_kernel, D = (X~ - X)^T X)",
                    "bound": "tensor", "achieved": a, "peak": burst, "unit": "TFLOP/s", "frac": a / burst,
                    "traffic": None, "peak_source": f"{peak_src} bf16 dense burst",
                    "algorithmic_flops_per_launch": fl["drift"], "executed_flops_per_launch": 2 * fl["drift"],
                    "executed_frac": 2 * a / burst, "syrk_h_x": roofline}

    e2e = None
    if not args.no_e2e:
        Xh = inp["X"].cpu().pin_memory()
        Xth = Xt.cpu().pin_memory() if drift else None
        Gh = inp["G"].cpu().pin_memory()
        Wh = inp["W"].cpu().pin_memory()
        suh, svh = inp["sign_u"].cpu().pin_memory(), inp["sign_v"].cpu().pin_memory()
        e2e_x = args.e2e_x_chunk_tokens
        if e2e_x is None:
            e2e_x = 32768 if cfg.T * cfg.d_in * 2 > (4 << 30) else args.x_chunk_tokens
        link = h2d_link_probe(dev)
        if args.e2e_g_chunk_tokens != args.g_chunk_tokens or e2e_x != args.x_chunk_tokens:
            p = LayerPipeline(cfg.d_out, cfg.d_in, cfg.bits, cfg.group, cfg.block, cfg.damp, device=dev,
                              x_chunk_tokens=e2e_x, g_chunk_tokens=args.e2e_g_chunk_tokens,
                              trailing=args.trailing, alpha=args.drift, drift_chunk_tokens=args.drift_chunk_tokens)
        ch = torch.empty(p.codes.shape, dtype=p.codes.dtype).pin_memory()
        sh = torch.empty(p.scale.shape, dtype=p.scale.dtype).pin_memory()
        zh = torch.empty(p.zero.shape, dtype=p.zero.dtype).pin_memory()
        p.run_host(Xh, Gh, Wh, suh, svh, ch, sh, zh, stream=stream, Xt_h=Xth)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier()
        torch.cuda.synchronize()
        e0.record(stream)
        nin = nout = 0
        e_steps = max(1, min(steps, 20))
        for _ in range(e_steps):
            nin, nout = p.run_host(Xh, Gh, Wh, suh, svh, ch, sh, zh, stream=stream, Xt_h=Xth)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        e_ms = max_over_ranks(e0.elapsed_time(e1), ws, dev)
        e2e = {"value": e_ms / (ws * e_steps), "unit": "ms", "h2d_bytes_per_step": nin,
               "d2h_bytes_per_step": nout, "steps": e_steps,
               "factor_chunk_tokens": {"X": e2e_x, "G": args.e2e_g_chunk_tokens}, "h2d_link": link,
               "bound_ms": max(total_ms / steps, nin / (max(link["gbs"].values()) * 1e6))}
        del Xh, Xth, Gh, Wh
    del p, inp, Xt, m
    torch.cuda.empty_cache()

    secondary = None
    if args.secondary and args.secondary != args.config and not drift and args.tokens == 0:
        scfg = kqsynth.CONFIGS[args.secondary].replace(seed=rank)
        ms = measure_layer(scfg, args, dev, ws, 50, stream, barrier, sample_clocks=False)
        secondary = {"workload": workload_name(scfg), "value": ms["total_ms"] / (ws * 50), "unit": "ms",
                     "steps": 50, "stages_ms": ms["stage_ms"], "gpu_launches": ms["launches"],
                     "fractions": fractions(scfg, ms["stage_ms"], peaks, peak_src)}
        del ms
        torch.cuda.empty_cache()

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = oracle_sample_ms(cfg, "large", alpha=args.drift)

    if rank == 0:
        out = {"metric": metric_of(args.drift), "value": total_ms / (ws * steps), "unit": "ms", "n_gpus": ws,
               "steps": steps, "warmup": args.warmup, "ms_per_step": total_ms / steps,
               "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
               "dtype": "bf16 products, f32 accumulate/arithmetic", "data": "synthetic",
               "config": config_dict(cfg, args.x_chunk_tokens, args.g_chunk_tokens, args.trailing, args.drift),
               "stages_ms": stage_ms, "tflops": tflops, "fractions": fractions(cfg, stage_ms, peaks, peak_src),
               "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches,
               "launch_mode": "cuda graph replay (one graph per layer, two streams)" if used_graph
               else "direct launches (two streams)",
               "clocks": clocks, "secondary": secondary}
        print(json.dumps(out), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


# ------------------------------------------------------------------ transformer block
BLOCK_METRIC = "ms per transformer block (7 sublayers: shared H_X, W2/W3 allocation, rotate+chol+sweep)"


def block_config_dict(bc, lanes) -> dict:
    return {"workload": (f"{bc.name}: d_model {bc.d_model}, d_kv {bc.d_kv}, d_ff {bc.d_ff}, T={bc.T} tokens, "
                         f"W{bc.low_bits}/W{bc.high_bits} at mean {bc.budget} bits, group {bc.group}"),
            "d_model": bc.d_model, "d_kv": bc.d_kv, "d_ff": bc.d_ff, "T": bc.T, "group": bc.group,
            "bits": [bc.low_bits, bc.high_bits], "budget_bits": bc.budget, "lanes": lanes,
            "l2": "inputs larger than L2 (every X and G is T x d bf16); no flush"}


def block_flops(bc) -> dict:
    spec = kqsynth.block_spec(bc)
    d_in = {grp: d for _, grp, _, d in spec}
    fx = sum(bc.T * d * (d + 1) for d in d_in.values())
    fg = sum(bc.T * d_out * (d_out + 1) for _, _, d_out, _ in spec)
    return {"factors": fx + fg, "factor_x": fx, "factor_g": fg}


def oracle_block_ms(bc, small: bool = False) -> dict:
    """The oracle's time for a block: the layer estimate of oracle_sample_ms per sublayer,
    minus the H_X accumulations the shared inputs do not repeat."""
    spec = kqsynth.block_spec(bc)
    preset = "medium" if small else "large"
    total, seen, parts = 0.0, set(), {}
    for name, grp, d_out, d_in in spec:
        c = kqsynth.LayerConfig(name, d_out, d_in, bc.T, bc.low_bits, bc.group, bc.n_outliers, bc.g_sigma,
                                block=bc.block, damp=bc.damp)
        r = oracle_sample_ms(c, preset, check=False)
        v = r["value"]
        if grp in seen:   # H_X of a shared input is accumulated once: drop this layer's X share
            v -= r["stages_ms"]["factors"] * d_in * d_in / (d_in * d_in + d_out * d_out)
        seen.add(grp)
        parts[name] = v
        total += v
    return {"value": total, "unit": "ms", "cores": os.cpu_count(), "kind": "oracle", "sublayers_ms": parts,
            "sample": "per sublayer the single-layer sample of oracle_sample_ms" + (" (reduced)" if small else "")
                      + "; shared H_X counted once"}


def run_block(args):
    import torch

    from paper_2607_07964_gb300 import build as kbuild
    ws, rank, local = dist_setup("nccl")
    kbuild.build()
    from paper_2607_07964_gb300 import kronq as kq
    from paper_2607_07964_gb300.block import BlockQuantizer

    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    bc = kqsynth.BLOCKS[args.block].replace(seed=rank)
    if args.tokens > 0:
        bc = bc.replace(T=args.tokens)
    spec = kqsynth.block_spec(bc)
    inp = kqsynth.device_block(bc, device=dev)
    q = BlockQuantizer(spec, bc.group, bc.block, bc.damp, bc.low_bits, bc.high_bits, bc.budget, device=dev,
                       trailing=args.trailing, lanes=args.lanes)
    stream = torch.cuda.current_stream()
    args_in = (inp["X"], inp["G"], inp["W"], inp["sign_u"], inp["sign_v"])
    for _ in range(args.warmup):
        q.run(*args_in, stream=stream)
    q.check()

    def barrier():
        if ws > 1:
            torch.distributed.barrier()

    sampler = ClockSampler(None)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    fac_ms, tot_ms = [], []
    barrier()
    torch.cuda.synchronize()
    sampler.start()
    n0 = kq.launch_count()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        ev[0].record(stream)
        q.factors(inp["X"], inp["G"], stream)
        ev[1].record(stream)
        sc = q.scores(inp["W"], stream)
        bits = q.allocate(sc)
        q.quantize(inp["W"], inp["sign_u"], inp["sign_v"], bits, stream)
        ev[2].record(stream)
        torch.cuda.synchronize()
        fac_ms.append(ev[0].elapsed_time(ev[1]))
        tot_ms.append(ev[0].elapsed_time(ev[2]))
    t1.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = kq.launch_count() - n0
    clocks = sampler.stop()
    q.check()
    total = max_over_ranks(t0.elapsed_time(t1), ws, dev)
    fl = block_flops(bc)
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    fac = statistics.mean(fac_ms)
    achieved = fl["factors"] / fac / 1e9
    roofline = {"kernel": "syrk_tc_kernel (the block's 4 H_X and 7 H_G accumulations, back to back)",
                "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": None, "peak_source": f"{peak_src} bf16 dense burst",
                "algorithmic_flops_per_launch": fl["factors"] / 11, "launches": 11}
    e2e = None
    if not args.no_e2e:
        hosts = {k: {n: t.cpu().pin_memory() for n, t in d.items()} for k, d in zip(
            ("X", "G", "W", "sign_u", "sign_v"), args_in)}
        outs = {n: (torch.empty(p.codes.shape, dtype=torch.uint8).pin_memory(),
                    torch.empty(p.scale.shape).pin_memory(), torch.empty(p.zero.shape, dtype=torch.int32).pin_memory())
                for n, p in q.pipes.items()}
        nin = sum(t.numel() * t.element_size() for d in hosts.values() for t in d.values())
        nout = sum(t.numel() * t.element_size() for o in outs.values() for t in o)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(args.steps):
            for key, d in hosts.items():
                for n, t in d.items():
                    args_in[("X", "G", "W", "sign_u", "sign_v").index(key)][n].copy_(t, non_blocking=True)
            q.run(*args_in, stream=stream)
            for n, (c, s_, z) in outs.items():
                p = q.pipes[n]
                c.copy_(p.codes, non_blocking=True)
                s_.copy_(p.scale, non_blocking=True)
                z.copy_(p.zero, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        e2e = {"value": max_over_ranks(e0.elapsed_time(e1), ws, dev) / (ws * args.steps), "unit": "ms",
               "h2d_bytes_per_step": nin, "d2h_bytes_per_step": nout,
               "note": "copies, then the block (no overlap of copies with compute)"}
    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = oracle_block_ms(bc)
    if rank == 0:
        out = {"metric": BLOCK_METRIC, "value": total / (ws * args.steps), "unit": "ms", "n_gpus": ws,
               "steps": args.steps, "warmup": args.warmup, "ms_per_step": total / args.steps,
               "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
               "dtype": "bf16 products, f32 accumulate/arithmetic", "data": "synthetic",
               "config": block_config_dict(bc, args.lanes),
               "stages_ms": {"factors": fac, "scores_alloc_quantize": statistics.mean(tot_ms) - fac},
               "bits": bits, "scores_post_biip": {n: sc[n][5] for n in sc},
               "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches // args.steps,
               "launch_mode": "direct launches; one host sync per block for the allocation", "clocks": clocks}
        print(json.dumps(out), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


# ------------------------------------------------------------------ decode (inference)
INFER_METRIC = "ms per decode step (B tokens through every linear sublayer, online BiIP revert)"


def run_infer(args):
    import torch

    from paper_2607_07964_gb300 import build as kbuild
    ws, rank, local = dist_setup("nccl")
    kbuild.build()
    from paper_2607_07964_gb300 import kronq as kq

    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    bc = kqsynth.BLOCKS["llama3_8b_block"]
    spec = kqsynth.block_spec(bc)
    bits, B, nb = args.infer, args.infer_tokens, args.infer_blocks
    gen = torch.Generator(device=dev)
    gen.manual_seed(1234 + rank)
    layers = []
    wbytes = 0
    for blk in range(nb):
        for name, _, d_out, d_in in spec:
            ng = d_in // 128
            codes = torch.randint(0, 2 ** bits, (d_out, d_in), generator=gen, device=dev, dtype=torch.int32).to(torch.uint8)
            packed = torch.empty(kq.kq_packed_codes_bytes(d_out, d_in, bits) // 4, dtype=torch.int32, device=dev)
            kq.kq_pack_codes(codes, bits, packed)
            del codes
            L = {"packed": packed, "d_out": d_out, "d_in": d_in,
                 "scale": torch.rand((d_out, ng), generator=gen, device=dev) * 0.01 + 1e-3,
                 "zero": torch.randint(0, 2 ** bits, (d_out, ng), generator=gen, device=dev, dtype=torch.int32),
                 "s_x": torch.rand(d_in, generator=gen, device=dev) + 0.5, "s_g": torch.rand(d_out, generator=gen, device=dev) + 0.5,
                 "su": (torch.randint(0, 2, (d_out,), generator=gen, device=dev) * 2 - 1).to(torch.int8),
                 "sv": (torch.randint(0, 2, (d_in,), generator=gen, device=dev) * 2 - 1).to(torch.int8)}
            L["x"] = torch.randn((B, d_in), generator=gen, device=dev)
            L["y"] = torch.empty((B, d_out), device=dev)
            L["ws"] = torch.empty(kq.kq_infer_workspace(B, d_in, d_out), dtype=torch.uint8, device=dev)
            wbytes += packed.numel() * 4 + L["scale"].numel() * 4 + L["zero"].numel() * 4
            layers.append(L)
    stream = torch.cuda.current_stream()
    # A block's decode step in dependency order, one stream: q, k, v, o, gate, up, down. Each
    # call's kernels launch as programmatic dependents of the ones before, so every layer's
    # weights head for L2 while the previous layer finishes.

    def call(L, s):
        kq.kq_infer(L["packed"], L["scale"], L["zero"], L["d_out"], L["d_in"], bits, 128, L["s_x"], L["s_g"],
                    L["su"], L["sv"], L["x"], L["y"], L["ws"], stream=s)

    def step(s):
        for L in layers:
            call(L, s)

    for _ in range(args.warmup):
        step(stream)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream(device=dev)
    n0 = kq.launch_count()
    with torch.cuda.graph(g, stream=cap):
        step(cap)
    per_step = kq.launch_count() - n0
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(None)
    sampler.start()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        g.replay()
    t1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = max_over_ranks(t0.elapsed_time(t1), ws, dev) / args.steps
    peaks, peak_src = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    ach = wbytes / ms / 1e6
    if rank == 0:
        out = {"metric": INFER_METRIC, "value": ms / ws, "unit": "ms", "n_gpus": ws, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": False, "scaling": "weak",
               "vs_baseline": None, "dtype": "f32 arithmetic on packed integer codes", "data": "synthetic",
               "config": {"workload": f"Llama-3-8B linear sublayers x {nb} blocks, {bits}-bit codes "
                                      f"({'4-bit lanes' if bits == 3 else 'packed'}), group 128, B = {B}; per block "
                                      f"q, k, v, o, gate, up, down in order on one stream",
                          "blocks": nb, "bits": bits, "tokens": B,
                          "l2": f"{wbytes / 1e9:.2f} GB of packed weights per step, larger than L2; no flush"},
               "roofline": {"kernel": "kq_infer (infer_stream_kernel + infer_out_kernel) over all sublayers",
                            "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
                            "traffic": None, "peak_source": f"{peak_src} HBM copy",
                            "bytes_per_step": wbytes},
               "cpu_baseline": None, "e2e": None, "gpu_launches": per_step,
               "launch_mode": "cuda graph replay", "clocks": clocks}
        print(json.dumps(out), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def run_validate(args):
    import torch

    from paper_2607_07964_gb300 import build as kbuild
    kbuild.build()
    from paper_2607_07964_gb300.validate import exponent_sweep

    cfg = kqsynth.CONFIGS[args.config]
    if args.tokens > 0:
        cfg = cfg.replace(T=args.tokens)
    inp = kqsynth.device_layer(cfg)
    alphas = [0.0, 0.125, 0.25, 0.375, 0.5]
    t0 = time.perf_counter()
    res = exponent_sweep(inp["X"], inp["G"], inp["W"], inp["sign_u"], inp["sign_v"], cfg.bits, cfg.group, alphas,
                         cfg.block, cfg.damp, args.trailing)
    wall = time.perf_counter() - t0
    base = res["loss"][alphas.index(0.25)]
    out = {"metric": "Prop. 2 output-side exponent sweep: proxy loss relative to alpha = 1/4",
           "config": config_dict(cfg, trailing=args.trailing), "data": "synthetic",
           "alphas": alphas, "loss": res["loss"], "loss_rel": [v / base for v in res["loss"]],
           "argmin_alpha": alphas[min(range(len(alphas)), key=lambda i: res["loss"][i])],
           "stats": res["stats"], "wall_s": wall}
    print(json.dumps(out), flush=True)


def main():
    args = parse()
    if args.validate:
        run_validate(args)
        return
    if args.infer is not None:
        run_infer(args)
        return
    if args.block is not None:
        if args.impl == "reference":
            ws, rank, _ = dist_setup("gloo")
            if rank == 0:
                bc = kqsynth.BLOCKS[args.block]
                if args.tokens > 0:
                    bc = bc.replace(T=args.tokens)
                t0 = time.perf_counter()
                vals = [oracle_block_ms(bc, small=True)["value"] for _ in range(args.steps)]
                v = statistics.mean(vals)
                print(json.dumps({"impl": "reference", "metric": BLOCK_METRIC, "value": v, "unit": "ms",
                                  "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                                  "ms_per_step": v, "higher_is_better": False, "scaling": "weak",
                                  "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                                  "config": block_config_dict(bc, args.lanes),
                                  "cpu_baseline": {"value": v, "unit": "ms", "cores": os.cpu_count(),
                                                   "kind": "oracle", "sample": "reduced single-layer samples"},
                                  "e2e": {"value": v, "unit": "ms", "h2d_bytes_per_step": 0,
                                          "d2h_bytes_per_step": 0},
                                  "wall_s": time.perf_counter() - t0}), flush=True)
        else:
            run_block(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
