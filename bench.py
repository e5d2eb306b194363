"""Benchmark: parameters decomposed + 2-bit coded per second at Llama-2-7B layer shapes.

One step = Algorithm 1 (k blocks) + closed-form centres + packed 2-bit codes for every
vector of one Llama-2-7B-shaped decoder layer (q, k, v, o: 4096x4096; gate, up:
4096x11008; down: 11008x4096 -- 202,375,168 parameters), through the C ABI
(kd_decompose, one call per matrix).  Steps cycle through the 32 layers of the
seeded 7B-shaped stack, generated once on the device and resident in HBM (13 GB
fp16), so no step re-reads an input another step touched; every input is larger
than L2.

Prints ONE JSON line on rank 0.  Extras in that line:
  roofline           ALU roofline of the dominant kernel (decompose at the length
                     carrying most parameters; N = 4096 for the 7B layer), measured
                     with CUDA events on the launch stream inside the timed region,
                     plus a measured FP32 peak and the FFT-count figure.
  cpu_baseline       the CPU oracle (fp64, dense DCT matrix) on a bounded sample.
  e2e                same metric with host (pinned) input buffers, H2D + D2H in the loop.
  clocks             nvidia-smi samples taken during the timed region.
  kmeans_refinement  cost of 3 Lloyd iterations of the centres (Sec. 2.1).
  hadamard_rotation  the Kashin-DCT+H pre-rotation of the layer, HBM roofline.
  inference_load     W_hat re-materialisation and factor expansion (App. C).

``--workload`` picks another synthetic stand-in per step (OPT-125M, Pythia-6.9B and
Mistral-7B-shaped layers, the single 256x256 matrix); ``--impl reference`` times the
CPU oracle instead (the reference arm).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "params decomposed+2-bit coded/sec at 7B layer shapes; % of roofline"
UNIT = "params/s"
ITERS = 16
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
PROFILE_FILE = os.path.join(ROOT, "profiles", "decompose_n4096_llama7b.json")


def _workloads():
    """Per-step workloads: name -> (number of seeded layers cycled, layer(L) -> specs,
    description).  The default is the Llama-2-7B layer; the others are the remaining
    synthetic stand-ins of the paper's models, for their own throughput lines."""
    from paper_2609_11687_gb300 import synth

    def fam(name):
        return lambda L: [s for s in synth.config5([L]) if s.name.startswith(name)]

    return {
        "llama7b": (32, synth.llama7b_layer,
                    "llama2-7b decoder layer per step: q,k,v,o 4096x4096, gate,up 4096x11008, down 11008x4096 "
                    "(202,375,168 params, fp16 Student-t nu=4 std 0.015, 0.1% input channels x20), cycling the "
                    "32 seeded layers of the 7B stack resident in HBM"),
        "w256": (1, lambda L: synth.config1(),
                 "one 256x256 fp32 matrix per step, 0.02 N(0,1), seed 0 (65,536 params)"),
        "opt125m": (12, lambda L: synth.config2([L]),
                    "OPT-125M-shaped layer per step: q,k,v,o 768x768, fc1 768x3072, fc2 3072x768 (7,077,888 "
                    "params, fp16 Student-t nu=4 std 0.02), cycling 12 seeded layers"),
        "pythia6.9b": (32, fam("pythia"),
                       "Pythia-6.9B-like layer per step: qkv 4096x12288, dense 4096x4096, h->4h 4096x16384, "
                       "4h->h 16384x4096 (201,326,592 params, fp16 Student-t nu=3 std 0.02, 0.05% entries x50), "
                       "cycling 32 seeded layers"),
        "mistral7b": (32, fam("mistral"),
                      "Mistral-7B-like layer per step: q,o 4096x4096, k,v 4096x1024, gate,up 4096x14336, down "
                      "14336x4096 (218,103,808 params, fp16 Student-t nu=3 std 0.02, 0.05% entries x50), cycling "
                      "32 seeded layers"),
    }
SM_COUNT = 152
L2_BYTES = 129 * 1024 * 1024
FP32_LANES_PER_SM = 128


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def flops_per_vector(n: int, iters: int) -> float:
    """Algorithmic FP32 work of Algorithm 1 on one vector (fixed convention):
    per block 4 length-n DCTs at 2 n log2 n each + 20 n for the four greedy steps."""
    return iters * (4 * 2 * n * math.log2(n) + 20 * n)


# sources the N = 4096 decompose kernel is built from (the profile's DRAM figures
# stay valid while these are unchanged)
DECOMPOSE_SOURCES = ("kd_math.cuh", "kd_xform.cuh", "kd_kernels.cuh", "kd_bulk.cuh", "kd_plans.cuh", "kd_launch.cuh", "kd_ops.h",
                     "kd_plan_4096.cu")


def fft_flops_per_vector(n: int, iters: int) -> float:
    """Secondary convention: 2.5 n log2 n per transform (the usual complex-FFT
    count), four transforms and 20 n greedy flops per block."""
    return iters * (4 * 2.5 * n * math.log2(n) + 20 * n)


def _code_only(text: str) -> str:
    """C++ source without comments and blank space: edits to comments do not
    change the kernel the profile figures were taken from."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_11687_gb300", "csrc")
    for name in DECOMPOSE_SOURCES:
        with open(os.path.join(csrc, name)) as f:
            h.update(name.encode())
            h.update(_code_only(f.read()).encode())
    return h.hexdigest()[:16]


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = sorted(float(r[1]) for r in rows if r[1].replace(".", "").isdigit())
        mx = max(float(r[2]) for r in rows if r[2].replace(".", "").isdigit())
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        power = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        return {"sm_mhz": sm[len(sm) // 2] if sm else None, "sm_max_mhz": mx, "reasons": reasons,
                "samples": len(rows), "power_w_max": max(power) if power else None}


# ---------------------------------------------------------------------------
# CPU oracle baseline (bounded sample)
# ---------------------------------------------------------------------------

_ORACLE_P = {}
ORACLE_SAMPLE_PARAMS = 1 << 17   # parameters per vector length in the fixed oracle sample


def oracle_sample(specs):
    """The fixed, seeded sample both CPU legs time (the GPU arm's cpu_baseline and the
    reference arm): per vector length n of the layer, the first 2 * round(2^16 / n)
    vectors (at least one pair, at most the matrix) of the first matrix of that length,
    drawn with that matrix's own seed.  Returns [(spec, x (n, m) float64)]."""
    import dataclasses
    from paper_2609_11687_gb300 import synth
    by_n = {}
    for s in specs:
        by_n.setdefault(s.N, s)
    out = []
    for n, spec in sorted(by_n.items()):
        m = max(2, 2 * round(ORACLE_SAMPLE_PARAMS / 2 / n))
        m = min(m, spec.M)
        G = synth.generate(dataclasses.replace(spec, M=m))
        out.append((spec, G.double().numpy().T.copy()))
    return out


def oracle_step(sample, iters: int, kmeans_iters: int = 0) -> dict:
    """One timed pass of the CPU oracle as it stands (decomposition, centres, codes,
    packing) over the fixed sample; the dense operator of each length is built once
    per process, outside the timed region.  Returns the per-length seconds."""
    from oracle import kashin_oracle as ko
    for spec, _ in sample:
        key = (spec.N, spec.sign_seed)
        if key not in _ORACLE_P:
            _ORACLE_P[key] = ko.POperator(spec.N, ko.sign_mask(spec.sign_seed, spec.N))
    secs = {}
    for spec, x in sample:
        P = _ORACLE_P[(spec.N, spec.sign_seed)]
        t0 = time.perf_counter()
        d = ko.decompose(x, P.eps, iters, P=P)
        cu = ko.centres(d.coeffs[0], d.coeffs[1])
        cv = ko.centres(d.coeffs[2], d.coeffs[3])
        if kmeans_iters:
            cu, code_u, _, _ = ko.kmeans_refine(d.u, cu, kmeans_iters)
            cv, code_v, _, _ = ko.kmeans_refine(d.vhat, cv, kmeans_iters)
        else:
            code_u, code_v = ko.codes(d.u, cu), ko.codes(d.vhat, cv)
        ko.pack_codes(code_u), ko.pack_codes(code_v)
        secs[spec.N] = time.perf_counter() - t0
    return secs


def oracle_rate(specs, sample, secs) -> float:
    """params/s of the whole layer mix from one step's per-length seconds (time per
    parameter measured per vector length, weighted by the layer's parameters there)."""
    per_param = {spec.N: secs[spec.N] / x.size for spec, x in sample}
    layer_params = sum(s.params for s in specs)
    return layer_params / sum(s.params * per_param[s.N] for s in specs)


def oracle_sample_desc(sample, iters, kmeans_iters) -> str:
    parts = ", ".join(f"{x.shape[1]} vectors of n={spec.N}" for spec, x in sample)
    return ("fp64 dense-DCT oracle, k=%d, kmeans=%d, on a fixed seeded sample (%s: the first vectors of the "
            "layer's first matrix of each length), scaled to the layer's parameter mix" % (iters, kmeans_iters, parts))


def oracle_baseline(specs, iters: int, kmeans_iters: int = 0, reps: int = 2) -> dict:
    """The CPU oracle timed on the fixed sample (best of `reps` passes after one
    untimed pass), as the GPU arm's cpu_baseline."""
    sample = oracle_sample(specs)
    oracle_step(sample, iters, kmeans_iters)            # untimed: operators, caches
    best = None
    for _ in range(reps):
        secs = oracle_step(sample, iters, kmeans_iters)
        v = oracle_rate(specs, sample, secs)
        best = v if best is None else max(best, v)
    return {"value": best, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": oracle_sample_desc(sample, iters, kmeans_iters)}


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def run_gpu(args) -> dict:
    import torch
    from paper_2609_11687_gb300 import build, synth

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    build.build()
    from paper_2609_11687_gb300 import kashin as kd

    iters = args.iters
    dev = torch.device("cuda", local)
    # this rank's layers: rank, rank + world, ...  (weak scaling, no data exchange)
    steps_total = args.warmup + args.steps
    from paper_2609_11687_gb300 import shard
    n_layers, layer_fn, workload_desc = _workloads()[args.workload]
    my_layers = shard.layer_schedule(rank, world, steps_total, n_layers)
    uniq = sorted(set(my_layers))
    log(f"[bench] rank {rank}/{world}: generating {len(uniq)} {args.workload} layers on {dev}")
    t0 = time.time()
    layers = {}
    for L in uniq:
        specs = layer_fn(L)
        layers[L] = [(s, synth.generate(s, device=dev)) for s in specs]
    torch.cuda.synchronize()
    log(f"[bench] generated in {time.time() - t0:.1f}s")
    layer_params = synth.total_params(layer_fn(0))
    # the dominant kernel: the vector length carrying most of the parameters
    by_n = {}
    for s_ in layer_fn(0):
        by_n[s_.N] = by_n.get(s_.N, 0) + s_.params
    NDOM = max(by_n, key=by_n.get)

    # outputs (one set per matrix of the layer) and workspaces, allocated once
    layer0 = layers[uniq[0]]
    outs = []
    for s, w in layer0:
        words = (s.N + 15) // 16
        outs.append(kd.Decomposed(
            codes_u=torch.empty((s.M, words), dtype=torch.int32, device=dev),
            codes_v=torch.empty((s.M, words), dtype=torch.int32, device=dev),
            centres_u=torch.empty((s.M, 4), dtype=torch.float32, device=dev),
            centres_v=torch.empty((s.M, 4), dtype=torch.float32, device=dev),
            coeffs=None, u=None, vhat=None, resid=None, trace=None))
    # matrices of one vector length go out in one kd_decompose_batch launch
    groups = {}
    for i, (s, _) in enumerate(layer0):
        groups.setdefault(s.N, []).append(i)
    wss = {n_: kd.Workspace(n_, dev) for n_ in groups}
    wsb = {n_: kd.Workspace(n_, dev, count=len(ix)) for n_, ix in groups.items()}
    stream = torch.cuda.current_stream()

    # kernels per step: batch = set-up + sign sets + decompose per length; single =
    # set-up + decompose per matrix (longer lengths always run one launch per matrix)
    if args.launch == "batch":
        launches_per_step = sum((3 if len(ix) > 1 else 2) if kd.kd_batchable(n_) else 2 * len(ix)
                                for n_, ix in groups.items())
    else:
        launches_per_step = 2 * len(layer0)
    ev_main = {}  # per-launch events of the dominant kernel
    ev_other = {}  # per-launch events of the other vector lengths' kernels

    def run_layer(L, record=False):
        mats = layers[L]
        for n_, ix in groups.items():
            rec = record
            if rec:
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
            if args.launch == "batch":
                kd.decompose_batch([mats[i][1] for i in ix], iters, [mats[i][0].sign_seed for i in ix],
                                   workspace=wsb[n_], outs=[outs[i] for i in ix], stream=stream,
                                   kmeans_iters=args.kmeans_iters)
            else:
                for i in ix:
                    kd.decompose(mats[i][1], iters, mats[i][0].sign_seed, workspace=wss[n_], out=outs[i],
                                 stream=stream, kmeans_iters=args.kmeans_iters)
            if rec:
                e1.record(stream)
                dst = ev_main.setdefault("ev", []) if n_ == NDOM else ev_other.setdefault(n_, [])
                dst.append((e0, e1, sum(mats[i][0].M for i in ix)))

    for i in range(args.warmup):
        run_layer(my_layers[i])
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    step_bytes = sum(w.numel() * w.element_size() for _, w in layers[uniq[0]])
    flush = None
    if step_bytes < 2 * L2_BYTES:
        # a step's input fits in L2: time each step alone and overwrite L2 between steps
        flush = torch.empty(4 * L2_BYTES // 4, dtype=torch.float32, device=dev)
        step_ms = 0.0
        for i in range(args.steps):
            flush.fill_(float(i))
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            run_layer(my_layers[args.warmup + i], record=True)
            b.record(stream)
            b.synchronize()
            step_ms += a.elapsed_time(b)
        l2_note = f"L2 overwritten between timed steps ({4 * L2_BYTES >> 20} MB write); steps timed one by one"
    else:
        start.record(stream)
        for i in range(args.steps):
            run_layer(my_layers[args.warmup + i], record=True)
        end.record(stream)
        l2_note = f"inputs larger than L2 ({step_bytes / 1e6:.0f} MB per step, distinct layer every step)"
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    clk = clocks.stop()
    elapsed_ms, total_params = shard.aggregate(step_ms if flush is not None else start.elapsed_time(end),
                                               args.steps * layer_params)
    value = total_params / (elapsed_ms / 1e3)
    del flush

    # dominant kernel: average launch duration over the timed region
    launches = ev_main.get("ev", [])
    dur = sum(a.elapsed_time(b) for a, b, _ in launches) / max(1, len(launches))
    vec_per_launch = sum(mm for _, _, mm in launches) / max(1, len(launches))
    fl = flops_per_vector(NDOM, iters) * vec_per_launch
    achieved_tflops = fl / (dur / 1e3) / 1e12
    peak = SM_COUNT * FP32_LANES_PER_SM * 2 * 2.070e9 / 1e12
    traffic = None
    if os.path.exists(PROFILE_FILE):
        with open(PROFILE_FILE) as f:
            prof = json.load(f)
        if prof.get("kernel_hash") == kernel_source_hash() and prof.get("iters") == iters and NDOM == 4096:
            traffic = prof["dram_bytes_per_vector"] * vec_per_launch
    roofline = {"bound": "alu", "achieved": round(achieved_tflops, 3), "peak": round(peak, 2),
                "unit": "TFLOP/s", "frac": round(achieved_tflops / peak, 4), "traffic": traffic,
                "kernel": f"decompose_kernel<N={NDOM}>", "launch_ms": round(dur, 3),
                "peak_basis": "FP32 FMA: 152 SMs x 128 lanes x 2 flop x 2070 MHz (max clock)"}
    if clk.get("sm_mhz"):
        roofline["frac_at_measured_clock"] = round(achieved_tflops / (peak * clk["sm_mhz"] / 2070.0), 4)
    # secondary: against a measured packed-FFMA peak of this GPU, and the work counted
    # with the conventional complex-FFT flop count (2.5 n log2 n per transform)
    meas = _extra(lambda: kd.measure_fp32_peak(stream))
    if isinstance(meas, float):
        roofline["measured_fp32_peak"] = round(meas, 2)
        roofline["frac_of_measured_fp32_peak"] = round(achieved_tflops / meas, 4)
    fl_fft = fft_flops_per_vector(NDOM, iters) * vec_per_launch
    roofline["achieved_fft_count"] = round(fl_fft / (dur / 1e3) / 1e12, 3)

    def other_kernels():
        out = []
        for n_, evs in sorted(ev_other.items()):
            d_ = sum(a.elapsed_time(b) for a, b, _ in evs) / len(evs)
            v_ = sum(mm for _, _, mm in evs) / len(evs)
            t_ = flops_per_vector(n_, iters) * v_ / (d_ / 1e3) / 1e12
            out.append({"kernel": f"decompose_kernel<N={n_}>", "launch_ms": round(d_, 3),
                        "achieved": round(t_, 3), "unit": "TFLOP/s", "frac": round(t_ / peak, 4)})
        return out
    if ev_other:
        roofline["other_kernels"] = _extra(other_kernels)

    # k-means refinement (Sec. 2.1): cost of KM_PROBE Lloyd iterations on the dominant
    # kernel, timed on the same matrices right after the timed region
    refinement = None
    if args.kmeans_iters == 0:
        refinement = _extra(lambda: measure_refinement(kd, torch, layers[my_layers[-1]], outs, wss, iters,
                                                       stream, NDOM))

    # randomized-Hadamard pre-rotation (Kashin-DCT+H), HBM roofline
    rotation = _extra(lambda: measure_rht(kd, torch, layers[my_layers[-1]], stream))
    # load-time inference expansion (App. C)
    inference = _extra(lambda: measure_inference(kd, torch, layers[my_layers[-1]], iters, wss, stream))

    # end to end: pinned host input, H2D + decompose + D2H codes/centres each step
    e2e = None
    if not args.skip_e2e:
        e2e = run_e2e(kd, torch, layers[uniq[0]], outs, wss, iters, args, stream, dist, world) if dist else \
            _extra(lambda: run_e2e(kd, torch, layers[uniq[0]], outs, wss, iters, args, stream, dist, world))

    result = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(elapsed_ms / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": workload_desc, "launch": args.launch,
                   "iters": iters, "kmeans_iters": args.kmeans_iters,
                   "layout": "vector-major (nn.Linear [out, in])",
                   "l2": l2_note,
                   "parallelism": f"dp{world} (layers sharded over ranks, no exchange)"},
        "roofline": roofline,
        "gpu_launches": args.steps * launches_per_step,
        "clocks": clk,
    }
    if refinement is not None:
        result["kmeans_refinement"] = refinement
    result["hadamard_rotation"] = rotation
    result["inference_load"] = inference
    if e2e is not None:
        result["e2e"] = e2e
    if rank == 0 and world == 1 and not args.skip_cpu:
        result["cpu_baseline"] = _extra(lambda: oracle_baseline(layer_fn(0), iters,
                                                 kmeans_iters=args.kmeans_iters))
    if dist:
        dist.destroy_process_group()
    return result if rank == 0 else None


KM_PROBE = 3
RHT_SEED = 0x5EED


def hbm_peak_gbs():
    if os.path.exists(PEAKS_FILE):
        with open(PEAKS_FILE) as f:
            v = json.load(f).get("hbm_gbs")
        if v:
            return float(v), "measured (MEASURED_PEAKS.json hbm_gbs, copy burst)"
    return 6800.0, "fallback 6.8 TB/s"


def _extra(fn):
    """Run one of the measurements reported beside the main figure; a failure there
    is reported in its place instead of losing the line."""
    try:
        return fn()
    except Exception as e:  # noqa: BLE001 -- any failure of an extra must not cost the main line
        log(f"[bench] extra measurement failed: {type(e).__name__}: {e}")
        return {"error": f"{type(e).__name__}: {e}"[:300]}


def measure_inference(kd, torch, layer, iters, wss, stream):
    """App. C at load time for one layer: dense W_hat = U_q + P V_q (kd_reconstruct,
    fp16 out; one P per vector pair, ALU-bound) and the two expanded factor planes
    for the folded product [X | XP][U_q; V_q] (kd_dequantise, fp16 out, HBM-bound)."""
    decs = [(s, kd.decompose(w, iters, s.sign_seed, workspace=wss[s.N], stream=stream)) for s, w in layer]
    # both factor planes of every matrix, grouped by vector length: one batched launch each
    groups = {}
    for s, d in decs:
        groups.setdefault(s.N, []).extend([(d.codes_u, d.centres_u), (d.codes_v, d.centres_v)])
    planes_out = {n: [torch.empty((c.shape[0], n), dtype=torch.float16, device=c.device) for c, _ in pl]
                  for n, pl in groups.items()}
    # a layer's code planes (about 0.1 GB) fit in L2: every repetition starts from a
    # flushed L2 (a 256 MB write outside the timed events); the median is reported
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=layer[0][1].device)

    def timed(fn, reps=6):
        evs = []
        for rep in range(reps):
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                flush.fill_(rep & 255)
            a.record(stream)
            fn()
            b.record(stream)
            if rep > 0:
                evs.append((a, b))
        torch.cuda.synchronize()
        ts = sorted(a.elapsed_time(b) for a, b in evs)
        return ts[len(ts) // 2]

    # every matrix to its own output, the matrices of one vector length in one launch
    rec_groups = {}
    for s, d in decs:
        rec_groups.setdefault(s.N, []).append((s, d, torch.empty((s.M, s.N), dtype=torch.float16,
                                                                 device=layer[0][1].device)))
    wsr = {n: kd.Workspace(n, layer[0][1].device, count=len(g)) for n, g in rec_groups.items()}

    def rec():
        for n, grp in rec_groups.items():
            kd.reconstruct_batch([d for _, d, _ in grp], n, [s.sign_seed for s, _, _ in grp], dtype=torch.float16,
                                 outs=[o for _, _, o in grp], workspace=wsr[n], stream=stream)

    def deq():
        for n, pl in groups.items():
            kd.dequantise_batch(pl, n, dtype=torch.float16, outs=planes_out[n], stream=stream)

    ms_rec = timed(rec)
    ms_deq = timed(deq)

    # the layer product straight from the 2-bit planes (one kd_matmul_2bit_batch for
    # the layer, XP from one kd_apply_p_prepared per vector length) against the dense fp16
    # product on the reconstructed W_hat (cuBLAS through torch.matmul), per batch of
    # activation rows
    dev = layer[0][1].device
    by_n = {}
    for k, (s_, _) in enumerate(decs):
        by_n.setdefault(s_.N, []).append(k)
    wsp = {n: kd.Workspace(n, dev, count=len(ix)) for n, ix in by_n.items()}
    folded = {}
    for bsz in (1, 4, 16):
        xs = {n: torch.randn((bsz, n), device=dev, dtype=torch.float32) for n in rec_groups}
        xps = [torch.empty_like(xs[s_.N]) for s_, _ in decs]
        ys = [torch.empty((bsz, s_.M), device=dev, dtype=torch.float32) for s_, _ in decs]
        x16 = {n: x.half() for n, x in xs.items()}

        def xp_tables_all():
            for n, ix in by_n.items():
                kd.apply_p_batch([xs[n]] * len(ix), [decs[k][0].sign_seed for k in ix], outs=[xps[k] for k in ix],
                                 workspace=wsp[n], stream=stream)

        # serving: P's tables derived once per layer (kd_prepare_p), then XP per batch
        prep = {n: kd.prepare_p(n, [decs[k][0].sign_seed for k in ix], stream=stream) for n, ix in by_n.items()}

        def xp_all():
            for n, ix in by_n.items():
                kd.apply_p_prepared([xs[n]] * len(ix), prep[n], outs=[xps[k] for k in ix], stream=stream)

        def prod_all():
            kd.matmul_2bit_batch([d for _, d in decs], [xs[s_.N] for s_, _ in decs], xps, outs=ys, stream=stream)

        def dense_all():
            with torch.cuda.stream(stream):
                for n, grp in rec_groups.items():
                    for _, _, wh in grp:
                        torch.matmul(x16[n], wh.T)

        # the tensor-core product for fp16 activations (X and XP rounded to fp16 by torch casts
        # outside the timed region, as the dense fp16 baseline's X is)
        xp_all()
        xp16 = [xp.half() for xp in xps]

        def prod16_all():
            kd.matmul_2bit_f16_batch([d for _, d in decs], [x16[s_.N] for s_, _ in decs], xp16, outs=ys,
                                     stream=stream)

        ms_xp, ms_prod, ms_dense = timed(xp_all, 6), timed(prod_all, 6), timed(dense_all, 6)
        ms_prod16, ms_xp_tables = timed(prod16_all, 6), timed(xp_tables_all, 6)
        code_bytes = sum(2 * s.M * ((s.N + 15) // 16) * 4 + 2 * s.M * 16 + bsz * s.M * 4 for s, _ in layer)
        prod_bytes = code_bytes + sum(2 * bsz * s.N * 4 for s, _ in layer)
        prod16_bytes = code_bytes + sum(2 * bsz * s.N * 2 for s, _ in layer)
        hbm_pk = hbm_peak_gbs()[0]
        folded[f"batch{bsz}"] = {
            "ms_product": round(ms_prod, 4), "ms_xp": round(ms_xp, 4), "ms_xp_deriving_tables": round(ms_xp_tables, 4),
            "ms_total": round(ms_prod + ms_xp, 4),
            "ms_dense_fp16": round(ms_dense, 4), "bound": "hbm",
            "achieved": round(prod_bytes / (ms_prod / 1e3) / 1e9, 1), "peak": hbm_pk, "unit": "GB/s",
            "frac": round(prod_bytes / (ms_prod / 1e3) / 1e9 / hbm_pk, 4),
            "f16_tc": {"ms_product": round(ms_prod16, 4), "ms_total": round(ms_prod16 + ms_xp, 4),
                       "vs_dense_fp16": round(ms_dense / ms_prod16, 2),
                       "achieved": round(prod16_bytes / (ms_prod16 / 1e3) / 1e9, 1), "peak": hbm_pk, "unit": "GB/s",
                       "frac": round(prod16_bytes / (ms_prod16 / 1e3) / 1e9 / hbm_pk, 4)}}
    params = sum(s.params for s, _ in layer)
    # one P (a DCT and an inverse DCT) per vector: 2 * 2 n log2 n flops, plus n adds
    import math
    flops = sum(s.M * (4 * s.N * math.log2(s.N) + s.N) for s, _ in layer)
    peak_alu = SM_COUNT * FP32_LANES_PER_SM * 2 * 2.070e9 / 1e12
    deq_bytes = 2 * params * (0.25 + 2)
    hbm, basis = hbm_peak_gbs()
    del planes_out
    return {
        "reconstruct": {"kernel": "reconstruct_kernel (codes -> fp16 W_hat, one kd_reconstruct_batch per vector "
                                  "length)",
                        "ms_per_layer": round(ms_rec, 4), "params_per_s": round(params / (ms_rec / 1e3), 1),
                        "bound": "alu", "achieved": round(flops / (ms_rec / 1e3) / 1e12, 3),
                        "peak": round(peak_alu, 2), "unit": "TFLOP/s",
                        "frac": round(flops / (ms_rec / 1e3) / 1e12 / peak_alu, 4)},
        "dequantise": {"kernel": "dequant_rows_batch_kernel (both planes of every matrix -> fp16, one "
                                 "batched launch per vector length: 2 per layer)",
                       "ms_per_layer": round(ms_deq, 4), "bound": "hbm",
                       "achieved": round(deq_bytes / (ms_deq / 1e3) / 1e9, 1), "peak": hbm, "unit": "GB/s",
                       "frac": round(deq_bytes / (ms_deq / 1e3) / 1e9 / hbm, 4), "peak_basis": basis,
                       "algorithmic_bytes_per_param": 4.5},
        "matmul_2bit": {"kernel": "fold_kernel (Y = X U_q^T + XP V_q^T from the 2-bit planes: one "
                                  "kd_matmul_2bit_batch per layer and group of up to 2 rows; XP by one "
                                  "kd_apply_p_prepared per vector length on tables kd_prepare_p derived once "
                                  "per layer; ms_xp_deriving_tables: kd_apply_p_batch, tables derived per call) "
                                  "against torch.matmul fp16 on W_hat "
                                  "(cuBLAS, one call per matrix), whole layer; f16_tc: fold16_kernel "
                                  "(kd_matmul_2bit_f16_batch, fp16 X and XP, mma.sync m16n8k16 with fp32 sums, "
                                  "one launch per 16 rows); L2 flushed before every repetition, median",
                        "algorithmic_bytes": "codes 0.5 B per weight + centres + x, XP, y", "peak_basis": basis,
                        **folded},
    }


def measure_rht(kd, torch, layer, stream):
    """Randomized-Hadamard rotation of the whole layer (Sec. 4, the Kashin-DCT+H
    preprocessing): fp16 in, fp32 out, one kd_rht per matrix, timed with events on
    the launch stream.  HBM-bound: 2 B read + 4 B written per parameter.  Reported
    per layer (seven launches back to back) and per launch (the largest matrix)."""
    # every matrix to its own output (outputs shared by equal shapes would let L2 absorb
    # part of the writes)
    outs = [torch.empty(tuple(w.shape), dtype=torch.float32, device=w.device) for _, w in layer]
    evs, big = [], []
    biggest = max(range(len(layer)), key=lambda i: layer[i][0].params)
    for rep in range(4):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i, (s, w) in enumerate(layer):
            if i == biggest:
                c = torch.cuda.Event(enable_timing=True)
                d = torch.cuda.Event(enable_timing=True)
                c.record(stream)
            kd.rht(w, RHT_SEED, out=outs[i], stream=stream)
            if i == biggest:
                d.record(stream)
                if rep > 0:
                    big.append((c, d))
        b.record(stream)
        if rep > 0:
            evs.append((a, b))
    torch.cuda.synchronize()
    ms = sum(a.elapsed_time(b) for a, b in evs) / len(evs)
    ms_big = sum(a.elapsed_time(b) for a, b in big) / len(big)
    params = sum(s.params for s, _ in layer)
    nbytes = params * (2 + 4)
    bytes_big = layer[biggest][0].params * 6
    peak, basis = hbm_peak_gbs()
    gbs = nbytes / (ms / 1e3) / 1e9
    gbs_big = bytes_big / (ms_big / 1e3) / 1e9
    del outs
    return {"kernel": "rht_staged_kernel (fp16 -> fp32, 7 launches per layer)", "ms_per_layer": round(ms, 4),
            "params_per_s": round(params / (ms / 1e3), 1), "bound": "hbm", "achieved": round(gbs, 1),
            "peak": peak, "unit": "GB/s", "frac": round(gbs / peak, 4), "peak_basis": basis,
            "algorithmic_bytes_per_param": 6,
            "largest_launch": {"matrix": layer[biggest][0].name, "ms": round(ms_big, 4),
                               "achieved": round(gbs_big, 1), "frac": round(gbs_big / peak, 4)}}


def measure_refinement(kd, torch, layer, outs, wss, iters, stream, ndom):
    """Cost of KM_PROBE Lloyd iterations on the dominant length: per-matrix launches
    of that length with and without the refinement, timed back to back."""
    def timed(km):
        evs = []
        for rep in range(3):
            for i, (s, w) in enumerate(layer):
                if s.N != ndom:
                    continue
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record(stream)
                kd.decompose(w, iters, s.sign_seed, workspace=wss[s.N], out=outs[i], stream=stream,
                             kmeans_iters=km)
                b.record(stream)
                if rep > 0:
                    evs.append((a, b))
        torch.cuda.synchronize()
        return sum(a.elapsed_time(b) for a, b in evs) / len(evs)
    base = timed(0)
    ms = timed(KM_PROBE)
    return {"kmeans_iters": KM_PROBE, "kernel": f"decompose_kernel<N={ndom}>", "launch_ms": round(ms, 3),
            "closed_form_launch_ms": round(base, 3), "overhead_vs_closed_form": round(ms / base - 1.0, 4)}


def run_e2e(kd, torch, layer, outs, wss, iters, args, stream, dist, world):
    """Same metric through the library's host-buffer entry point: every step, for
    each vector length, one kd_decompose_batch_host call uploads that group's fp16
    weights from pinned host memory, decomposes them in one batched launch and reads
    the codes and centres back into pinned host memory, all on one stream.  Two slots
    per group (stream, device staging, workspace, host outputs) alternate between
    steps, so one step's copies overlap the other slot's decomposition."""
    host_in = [(s, w.cpu().pin_memory()) for s, w in layer]
    groups = {}
    for i, (s, _) in enumerate(layer):
        groups.setdefault(s.N, []).append(i)
    slots = {}
    for n_, ix in groups.items():
        ws_h = [host_in[i][1] for i in ix]
        nbytes = kd.staging_size_host(ws_h)
        slots[n_] = [{"stream": torch.cuda.Stream(device=stream.device),
                      "staging": torch.empty(nbytes, dtype=torch.uint8, device=stream.device),
                      "ws": kd.Workspace(n_, stream.device, count=len(ix)),
                      "outs": [kd.host_outputs(host_in[i][1].shape[0], n_) for i in ix]} for _ in range(2)]
    h2d = sum(w.numel() * w.element_size() for _, w in host_in)
    d2h = sum(t.numel() * t.element_size() for o in outs for t in (o.codes_u, o.codes_v, o.centres_u, o.centres_v))
    count = [0]

    def step():
        k = count[0] % 2
        count[0] += 1
        for n_, ix in groups.items():
            sl = slots[n_][k]
            kd.decompose_batch_host([host_in[i][1] for i in ix], iters, [host_in[i][0].sign_seed for i in ix],
                                    sl["outs"], sl["staging"], sl["ws"], stream=sl["stream"],
                                    kmeans_iters=args.kmeans_iters)

    all_streams = [sl["stream"] for v in slots.values() for sl in v]
    for _ in range(2):
        step()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    n = max(5, args.steps)
    a.record(stream)
    for st in all_streams:
        st.wait_event(a)
    for _ in range(n):
        step()
    for st in all_streams:
        e = torch.cuda.Event()
        e.record(st)
        stream.wait_event(e)
    b.record(stream)
    torch.cuda.synchronize()
    # the host copies of the last step equal a device-resident run of the same layer
    last = (count[0] - 1) % 2
    for n_, ix in groups.items():
        ref = kd.decompose_batch([host_in[i][1].to(stream.device) for i in ix], iters,
                                 [host_in[i][0].sign_seed for i in ix], stream=stream, kmeans_iters=args.kmeans_iters)
        torch.cuda.synchronize()
        for r, o in zip(ref, slots[n_][last]["outs"]):
            if not (torch.equal(o.codes_u, r.codes_u.cpu()) and torch.equal(o.centres_v, r.centres_v.cpu())):
                raise RuntimeError("e2e host outputs differ from the device-resident run")
    from paper_2609_11687_gb300 import shard
    params = sum(s.params for s, _ in layer)
    ms, total = shard.aggregate(a.elapsed_time(b), n * params)
    return {"value": round(total / (ms / 1e3), 1), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": n,
            "pipeline": "kd_decompose_batch_host per vector length (H2D from pinned host memory, one batched "
                        "decompose, D2H of codes and centres, all on one stream), two alternating slots per "
                        "length on their own streams"}


# ---------------------------------------------------------------------------
# reference arm: the CPU oracle as it stands
# ---------------------------------------------------------------------------

def run_reference(args) -> dict | None:
    """The reference arm: the CPU oracle as it stands on the host cores.  Every step
    is one pass over the same fixed seeded sample the GPU arm's cpu_baseline times;
    ms_per_step is that pass's wall time, value the layer-mix params/s it gives
    (mean over the timed steps)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return None
    _, layer_fn, workload_desc = _workloads()[args.workload]
    specs = layer_fn(0)
    sample = oracle_sample(specs)
    oracle_step(sample, args.iters, args.kmeans_iters)   # builds the operators (not a step)
    rates, walls = [], []
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        secs = oracle_step(sample, args.iters, args.kmeans_iters)
        wall = time.perf_counter() - t0
        if i >= args.warmup:
            rates.append(oracle_rate(specs, sample, secs))
            walls.append(wall)
    value = sum(rates) / len(rates)
    sample_params = sum(x.size for _, x in sample)
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": int(os.environ.get("WORLD_SIZE", "1")), "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": sum(walls) / len(walls) * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc + "; each step one pass of the CPU oracle over a fixed seeded "
                               "sample of that layer (%d parameters) on the host cores, scaled to the layer's "
                               "parameter mix" % sample_params, "iters": args.iters,
                   "kmeans_iters": args.kmeans_iters, "sample_params_per_step": sample_params},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                         "sample": oracle_sample_desc(sample, args.iters, args.kmeans_iters)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def run_profile_case(args) -> None:
    """Small case for ncu: one matrix of the workload's layer with M vectors (default
    the 7B layer's q: n = 4096, M = 32768, 256 MB of input, above L2), decomposed 3
    times."""
    import dataclasses
    import torch
    from paper_2609_11687_gb300 import build, synth
    build.build()
    from paper_2609_11687_gb300 import kashin as kd
    layer_fn = _workloads()[args.workload][1]
    spec = dataclasses.replace(layer_fn(0)[args.profile_matrix], M=args.profile_m)
    w = synth.generate(spec, device="cuda")
    if args.profile_kernel in ("reconstruct", "dequantise"):
        dec = kd.decompose(w, args.iters, spec.sign_seed)
        y = torch.empty(w.shape, dtype=torch.float16, device="cuda")
        for _ in range(3):
            if args.profile_kernel == "reconstruct":
                kd.reconstruct(dec, spec.N, spec.sign_seed, dtype=torch.float16, out=y)
            else:
                kd.dequantise(dec.codes_u, dec.centres_u, spec.N, out=y)
        torch.cuda.synchronize()
        log(f"[profile-case] ok: {args.profile_kernel} n={spec.N} m={spec.M}")
        return
    if args.profile_kernel == "fold":
        # the layer's 2-bit products at batch 1 (one kd_matmul_2bit_batch), three times
        decs = []
        for s_ in layer_fn(0):
            w_ = synth.generate(s_, device="cuda")
            decs.append((s_, kd.decompose(w_, args.iters, s_.sign_seed)))
            del w_
        xs = {n: torch.randn((1, n), device="cuda") for n in {s_.N for s_, _ in decs}}
        xps = [kd.apply_p(xs[s_.N], s_.sign_seed) for s_, _ in decs]
        for _ in range(3):
            kd.matmul_2bit_batch([d for _, d in decs], [xs[s_.N] for s_, _ in decs], xps)
        torch.cuda.synchronize()
        log("[profile-case] ok: fold, 7B layer, batch 1")
        return
    if args.profile_kernel == "fold16":
        # the layer's fp16 tensor-core products at batch 4 (one kd_matmul_2bit_f16_batch), three times
        decs = []
        for s_ in layer_fn(0):
            w_ = synth.generate(s_, device="cuda")
            decs.append((s_, kd.decompose(w_, args.iters, s_.sign_seed)))
            del w_
        xs = {n: torch.randn((4, n), device="cuda") for n in {s_.N for s_, _ in decs}}
        xps = [kd.apply_p(xs[s_.N], s_.sign_seed).half() for s_, _ in decs]
        x16 = {n: x.half() for n, x in xs.items()}
        for _ in range(3):
            kd.matmul_2bit_f16_batch([d for _, d in decs], [x16[s_.N] for s_, _ in decs], xps)
        torch.cuda.synchronize()
        log("[profile-case] ok: fold16, 7B layer, batch 4")
        return
    if args.profile_kernel == "rht":
        y = torch.empty(w.shape, dtype=torch.float32, device="cuda")
        for _ in range(3):
            kd.rht(w, RHT_SEED, out=y)
        torch.cuda.synchronize()
        log(f"[profile-case] ok: rht n={spec.N} m={spec.M}")
        return
    ws = kd.Workspace(spec.N)
    out = None
    for _ in range(3):
        out = kd.decompose(w, args.iters, spec.sign_seed, workspace=ws, out=out, kmeans_iters=args.kmeans_iters)
    torch.cuda.synchronize()
    log(f"[profile-case] ok: n={spec.N} m={spec.M} iters={args.iters} kmeans={args.kmeans_iters}")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=32)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--iters", type=int, default=ITERS)
    ap.add_argument("--kmeans-iters", type=int, default=0,
                    help="Lloyd refinement iterations of the centres (Sec. 2.1); 0 = closed form")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--launch", default="batch", choices=["batch", "single"],
                    help="one kd_decompose_batch launch per vector length (default) or one launch per matrix")
    ap.add_argument("--workload", default="llama7b",
                    choices=["llama7b", "w256", "opt125m", "pythia6.9b", "mistral7b"],
                    help="synthetic stand-in per step (default: one Llama-2-7B-shaped layer)")
    ap.add_argument("--skip-cpu", action="store_true")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--profile-case", action="store_true", help="small single-matrix case for ncu")
    ap.add_argument("--profile-m", type=int, default=32768)
    ap.add_argument("--profile-matrix", type=int, default=0, help="layer matrix index (0 = q, 6 = down)")
    ap.add_argument("--profile-kernel", default="decompose", choices=["decompose", "rht", "reconstruct", "dequantise", "fold", "fold16"])
    args = ap.parse_args()
    if args.profile_case:
        run_profile_case(args)
        return
    if args.warmup < 3:
        log("[bench] warmup raised to 3 (timing rule)")
        args.warmup = 3
    res = run_reference(args) if args.impl == "reference" else run_gpu(args)
    if res is not None:
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
