"""Benchmark of one 1-bit FQT layer training step (forward + AGP/SCQ backward).

Metric: effective TOPS = 6 M K D (dense-equivalent operations of the forward,
grad_input and grad_weight products) / device time of the whole step, on the
ResNet-18 (CIFAR) 3x3 conv 256->256 layer on 8x8 maps, batch 128
(M = 8192, K = 2304, D = 256; AGP b = 4, keep 1/4 of samples and channels).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl fqt1|reference]

Each GPU runs an independent replica of the step (weak scaling; the layer step
has no exchange).  The step is captured once in a CUDA graph and replayed; L2
is flushed (256 MiB write) before every timed step and each step is timed with
CUDA events on the launching stream.  One JSON line is printed by rank 0.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "effective TOPS of 1-bit FQT layer fwd+bwd step; % of INT8 TC peak / HBM BW"
UNIT = "TOPS"
WORKLOAD = "resnet18-cifar conv3x3 256->256 8x8 batch128 (M=8192 K=2304 D=256), AGP b4 keep 1/4, SCQ"
# Peak used when MEASURED_PEAKS.json is absent.
FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS = 6800.0, 1900.0
SMS, POPC_PER_CLK_SM = 152, 16

# DRAM bytes (read + write) per launch of each stage's kernels, from one ncu capture of
# `bench.py --profile 2 --warmup 1` (the SCQ stage is the sum of its range, selection and
# quantize kernels).  A figure is valid only for
# the kernel sources it was taken on: TRAFFIC_SOURCES holds, per stage, the sha256 prefix of the
# files that define that stage's kernels (STAGE_SOURCES) at the capture; a stage whose sources
# have changed since reports traffic = null.
STAGE_SOURCES = {"pack": ("common.cuh", "pack.cu"), "gemm": ("api.cu", "common.cuh", "gemm.cuh", "gemm_tc.cu"),
                 "scq": ("common.cuh", "quantize.cu")}
STAGE_GROUP = {"pack_w": "pack", "pack_xp": "pack", "im2col": "pack", "fwd_gemm": "gemm", "scq_quantize": "scq",
               "bwd_input_fold": "gemm", "bwd_weight_gemm": "gemm"}
TRAFFIC_SOURCES = {"pack": "152daac4263996dc", "gemm": "59e795348d529633", "scq": "42a74653e8857164"}
TRAFFIC_BYTES = {"pack_w": 2.383872e+06, "im2col": 8.423680e+06, "fwd_gemm": 3.029504e+06,
                 "scq_quantize": 1.6950016e+07, "bwd_input_fold": 1.205504e+06,
                 "bwd_weight_gemm": 2.982144e+06}


def sources_sha(group):
    """sha256 prefix of the kernel sources of one stage group (file names and contents)."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2408_14267_gb300", "csrc")
    for f in sorted(STAGE_SOURCES[group]):
        h.update(f.encode())
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def stage_traffic(stage):
    g = STAGE_GROUP.get(stage)
    if g is None or stage not in TRAFFIC_BYTES or sources_sha(g) != TRAFFIC_SOURCES.get(g):
        return None
    return TRAFFIC_BYTES[stage]

CPU_SAMPLE_SCRIPT = r"""
import json, sys, time
sys.path.insert(0, sys.argv[1])
from paper_2408_14267_gb300 import workloads as wl
from oracle import method as om
w = wl.resnet18_cifar_conv()
batch, steps = int(sys.argv[2]), int(sys.argv[3])
first = int(sys.argv[4]) if len(sys.argv) > 4 else 0
N, C, H, W = w["x"].shape
Ho = Wo = H
x = w["x"][first:first + batch]
gy = w["gy"][first * Ho * Wo:(first + batch) * Ho * Wo]
def step():
    om.layer_step_conv(x, w["w"], w["gamma"], gy, w["stride"], w["pad"], w["bits_s"], w["mode_s"], w["seed_s"],
                       w["bits_c"], w["mode_c"], w["seed_c"])
if len(sys.argv) > 5:  # one untimed step, then start together with the other processes
    step()
    print("ready", flush=True)
    sys.stdin.readline()
times = []
t_start = time.time()
for _ in range(steps):
    t0 = time.perf_counter()
    step()
    times.append(time.perf_counter() - t0)
t_end = time.time()
M, K, D = batch * Ho * Wo, C * 9, w["w"].shape[0]
print(json.dumps({"times": times, "ops": 6.0 * M * K * D, "M": M, "K": K, "D": D, "t_start": t_start,
                  "t_end": t_end}))
"""


def run_oracle_sample(batch, steps):
    """Time the CPU oracle (as it stands) on `batch` samples of the workload, one thread."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               NUMEXPR_NUM_THREADS="1")
    p = subprocess.run([sys.executable, "-c", CPU_SAMPLE_SCRIPT, ROOT, str(batch), str(steps)], env=env,
                       capture_output=True, text=True, timeout=1800)
    if p.returncode != 0:
        raise RuntimeError("oracle sample failed: " + p.stderr[-2000:])
    return json.loads(p.stdout.strip().splitlines()[-1])


def host_cores():
    """Cores this process may run on: its CPU affinity, capped by a cgroup v2 CPU quota."""
    n = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    try:
        with open("/sys/fs/cgroup/cpu.max") as f:
            quota, period = f.read().split()[:2]
        if quota != "max":
            n = min(n, max(1, int(quota) // int(period)))
    except (OSError, ValueError):
        pass
    return n


def run_oracle_parallel(batch, procs, steps=1):
    """The oracle on `procs` host cores at once: one single-threaded process per core, each on
    its own slice of `batch` samples, all started together once every process has drawn its
    inputs.  Throughput = all processes' operations / (last end - first start)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               NUMEXPR_NUM_THREADS="1")
    ps = [subprocess.Popen([sys.executable, "-c", CPU_SAMPLE_SCRIPT, ROOT, str(batch), str(steps),
                            str((i * batch) % 128), "together"], env=env, stdin=subprocess.PIPE,
                           stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True) for i in range(procs)]
    try:
        for p in ps:
            if p.stdout.readline().strip() != "ready":
                raise RuntimeError("oracle process failed: " + p.stderr.read()[-2000:])
        for p in ps:
            p.stdin.write("go\n")
            p.stdin.flush()
        outs = [p.communicate(timeout=1800) for p in ps]
    finally:
        for p in ps:
            if p.poll() is None:
                p.kill()
                p.wait()
    rs = []
    for p, (out, err) in zip(ps, outs):
        if p.returncode != 0:
            raise RuntimeError("oracle process failed: " + err[-2000:])
        rs.append(json.loads(out.strip().splitlines()[-1]))
    wall = max(r["t_end"] for r in rs) - min(r["t_start"] for r in rs)
    ops = sum(r["ops"] * len(r["times"]) for r in rs)
    return {"value": ops / wall / 1e12, "cores": procs, "wall_s": wall, "M": rs[0]["M"], "K": rs[0]["K"],
            "D": rs[0]["D"]}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d.get("hbm_gbs", FALLBACK_HBM_GBS), d.get("bf16_tflops", FALLBACK_BF16_TFLOPS), "measured"
    return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons, sampled every 100 ms while running."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        # the raw samples go to FQT1_CLOCKS_DIR (default: the system temporary directory)
        import tempfile
        out_dir = os.environ.get("FQT1_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out_dir, f"clocks_gpu{gpu_index}.csv")

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            self.proc.wait(timeout=10)
            self.f.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


def max_over_ranks(x, device="cpu"):
    """The largest x over all ranks of the default process group (x itself without one).

    Replicas time their own K steps; the job took as long as its slowest rank."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tops(ops_per_step, steps, world, total_ms):
    """Whole-job throughput (tera-ops/s): each of `world` replicas ran `steps` steps of
    `ops_per_step` operations, and the slowest rank needed `total_ms`."""
    return world * ops_per_step * steps / (total_ms * 1e-3) / 1e12


def stage_work(st, name):
    """Algorithmic work of one stage: ('hbm', bytes) or ('tensor', dense-equivalent operations).

    The products run on e4m3 tensor cores, so their peak is the fp8 dense rate (twice the
    measured bf16 rate, the nominal ratio)."""
    from paper_2408_14267_gb300 import fqt1
    M, K, D = st.M, st.K, st.D
    wK, wM, wD = fqt1.packed_words(K), fqt1.packed_words(M), fqt1.packed_words(D)
    ks = st.psq.count() * st.rpg
    kc = st.pcq.count()
    if name == "pack_w":
        return "hbm", D * K * 4 + (D * wK + K * wD + K) * 4
    if name in ("im2col", "pack_x"):
        return "hbm", st.x.numel() * 4 + (M * wK + K * wM + K) * 4
    if name == "fwd_gemm":
        return "tensor", 2.0 * M * K * D
    if name == "scq_quantize":
        return "hbm", M * D * 4 + ks * D + kc * M
    if name in ("bwd_input_gemm", "bwd_input_fold"):
        return "tensor", 2.0 * ks * D * K
    if name == "col2im":
        return "hbm", ks * K * 4 + st.dx.numel() * 4
    if name == "bwd_weight_gemm":
        return "tensor", 2.0 * kc * M * K
    return "hbm", 0


def stage_times(st, stream, flush, reps):
    """Mean device time (ms) of each stage of the step, eager: the L2 is flushed, a sleep kernel
    holds the stream while all launches are queued, and CUDA events on the launching stream
    bracket every stage."""
    import torch
    stages = st.stages()
    per_stage = {n: [] for n, _ in stages}
    with torch.cuda.stream(stream):
        for _ in range(reps):
            flush.zero_()
            torch.cuda._sleep(2_000_000)
            evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)]
            evs[0].record(stream)
            for i, (n, fn) in enumerate(stages):
                fn(stream)
                evs[i + 1].record(stream)
            stream.synchronize()
            for i, (n, _) in enumerate(stages):
                per_stage[n].append(evs[i].elapsed_time(evs[i + 1]))
    return {n: statistics.mean(v) for n, v in per_stage.items()}


GEMM_STAGES = (("fwd", ("fwd_gemm",)), ("bwd_input", ("bwd_input_fold", "bwd_input_gemm")),
               ("bwd_weight", ("bwd_weight_gemm",)))


def gemm_rooflines(st, stage_ms, bf16_peak, peak_src):
    """Tensor roofline of each of the three products: algorithmic operations (2 M K D for the
    forward, 2 (kept rows) D K for grad_input, 2 (kept channels) M K for grad_weight) over the
    stage's device time, against the fp8 dense peak (2 x the bf16 peak: the nominal fp8/bf16
    ratio; the products run on e4m3 tensor cores)."""
    out = {}
    peak = 2.0 * bf16_peak
    for key, names in GEMM_STAGES:
        name = next((n for n in names if n in stage_ms), None)
        if name is None:
            continue
        _, ops = stage_work(st, name)
        us = stage_ms[name] * 1e3
        tf = ops / (us * 1e-6) / 1e12
        out[key] = {"kernel_stage": name, "ops": ops, "time_us": round(us, 3), "achieved": round(tf, 2),
                    "peak": peak, "unit": "TFLOP/s", "frac": tf / peak,
                    "peak_note": f"fp8 dense = 2 x {peak_src} bf16 (nominal fp8/bf16 ratio)"}
        if name == "bwd_input_fold":
            out[key]["note"] = "the Folder and the dequantization run in the same kernel's epilogue"
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="fqt1", choices=["fqt1", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--implicit", action="store_true",
                    help="implicit-GEMM forward (pixel-major sign(X), no unfolded row packing)")
    ap.add_argument("--e4m3-weights", choices=["on", "off"], default="on",
                    help="e4m3 copies of sign(W) written by the weight packing and loaded by TMA as the "
                         "B operand of the forward and grad_input products")
    ap.add_argument("--e4m3-x", choices=["on", "off"], default="off",
                    help="e4m3 copies of sign(X_u) written by the Unfolder and loaded by TMA as the sign "
                         "operand of the forward and grad_weight products")
    ap.add_argument("--profile", type=int, default=0, metavar="N",
                    help="only run --warmup + N eager steps (for ncu), print nothing")
    ap.add_argument("--profile-layer", metavar="NAME",
                    help="with --profile: the eager steps run this layer of the --layers sweep instead "
                         "(e.g. resnet18.stem, resnet18.layer1, vgg16.conv2)")
    ap.add_argument("--table5", action="store_true",
                    help="GEMM-only comparison of average 1-bit and 1-bit products on the Table 5 shapes")
    ap.add_argument("--model", choices=["vgg16", "resnet18"],
                    help="training step of a synthetic model built from binop layers against FP32 PyTorch")
    ap.add_argument("--layers", choices=["vgg16", "resnet18", "all"],
                    help="the layer step on every VGG-16 / ResNet-18 layer shape")
    ap.add_argument("--colmajor", choices=["auto", "on", "off"], default="auto",
                    help="--layers: grad_input of convolutions without the fused Folder through column-major "
                         "int32 accumulators and the column-major Folder (auto: the library's default)")
    ap.add_argument("--variance", action="store_true",
                    help="empirical variance of the AGP quantizer (b = 2, 4, 8) and of 1-bit PSQ against Eq. 24")
    ap.add_argument("--sweep", choices=["routine", "diag", "full"],
                    help="GEMM-shaped layer sweep: routine = M=D=K=4096, 256 groups, b = 1, 2, 4, 8; "
                         "diag = M=D=K in 1024..16384, 256 groups, b = 4; full = the whole grid")
    ap.add_argument("--res", type=int, default=32, help="input resolution of --model")
    ap.add_argument("--batch", type=int, default=128, help="batch of --model")
    args = ap.parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        return reference_arm(args, world, rank)
    if args.table5:
        return table5(args)
    if args.model:
        return model_step(args)
    if args.variance:
        return variance_study(args)
    if args.layers:
        return layer_sweep(args)
    if args.sweep:
        return gemm_sweep(args)

    import torch
    import torch.distributed as dist
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local_rank)
    from paper_2408_14267_gb300 import build, fqt1, workloads
    if rank == 0 or world == 1:
        build.build()
    if world > 1:
        dist.barrier()
    from paper_2408_14267_gb300.layer import LayerStep

    wl = workloads.resnet18_cifar_conv()
    if args.profile and args.profile_layer:  # another layer shape of the sweep, for ncu
        named = {w["name"].split()[0]: w for w in workloads.vgg16_layers(bits=4) + workloads.resnet18_imagenet_layers()}
        if args.profile_layer not in named:
            raise SystemExit(f"--profile-layer: one of {sorted(named)}")
        wl = named[args.profile_layer]
    st = LayerStep(wl, device=f"cuda:{local_rank}", keep_acc=False, implicit=args.implicit,
                   e4m3_weights=args.e4m3_weights == "on", e4m3_x=args.e4m3_x == "on")
    stream = torch.cuda.Stream()
    if args.profile:
        # eager steps, each after an L2 flush as in the timed loop (with ncu --cache-control none
        # the counters then show the step's own DRAM traffic)
        flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")
        with torch.cuda.stream(stream):
            for _ in range(args.warmup + args.profile):
                flush.zero_()
                st.step()
        torch.cuda.synchronize()
        return
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")  # 256 MiB > 129 MB L2
    with torch.cuda.stream(stream):
        for _ in range(max(args.warmup, 3)):
            st.step()
        stream.synchronize()
        n0 = fqt1.kernel_launches()
        st.step()
        stream.synchronize()
        launches_per_step = fqt1.kernel_launches() - n0
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            st.step_concurrent(stream)
        for _ in range(args.warmup):
            graph.replay()
        stream.synchronize()

    def timed_loop(k, sampler_steps=0):
        times = []
        with torch.cuda.stream(stream):
            for i in range(k):
                flush.zero_()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                graph.replay()
                e1.record(stream)
                times.append((e0, e1))
            stream.synchronize()
        return [a.elapsed_time(b) for a, b in times]

    # steady-state pre-roll so that the clock samples bracket a loaded GPU
    with ClockSampler(local_rank) as clk:
        t_end = time.time() + 0.8
        while time.time() < t_end:
            timed_loop(20)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        step_ms = timed_loop(args.steps)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        t_end = time.time() + 0.3
        while time.time() < t_end:
            timed_loop(20)
    clocks = clk.summary()
    total_ms = max_over_ranks(sum(step_ms), "cuda")
    ms_per_step = total_ms / args.steps
    ops = st.dense_ops()
    value = job_tops(ops, args.steps, world, total_ms)

    # per-stage device time (eager; the stream is held by a sleep kernel while all launches are queued)
    stage_ms = stage_times(st, stream, flush, max(10, min(args.steps, 50)))
    dom = max(stage_ms, key=stage_ms.get)
    hbm_peak, bf16_peak, peak_src = load_peaks()
    bound, work = stage_work(st, dom)
    dur_s = stage_ms[dom] * 1e-3
    if bound == "hbm":
        roof = {"bound": "hbm", "achieved": work / dur_s / 1e9, "peak": hbm_peak, "unit": "GB/s"}
    elif bound == "tensor":
        roof = {"bound": "tensor", "achieved": work / dur_s / 1e12, "peak": 2.0 * bf16_peak, "unit": "TFLOP/s",
                "peak_note": "fp8 dense = 2 x measured bf16 (nominal fp8/bf16 ratio)"}
    else:
        clk_mhz = clocks.get("sm_max_mhz") or 2070.0
        alu_peak = SMS * POPC_PER_CLK_SM * 32 * 2 * clk_mhz * 1e6 / 1e12
        roof = {"bound": "alu", "achieved": work / dur_s / 1e12, "peak": alu_peak, "unit": "TOPS"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = stage_traffic(dom)
    roof["kernel"] = dom
    roof["peak_source"] = peak_src if bound != "alu" else "derived: 152 SMs x 16 popc/clk x 32 bit x 2 x max clock"
    roof["gemms"] = gemm_rooflines(st, stage_ms, bf16_peak, peak_src)

    # end to end: pinned host inputs -> device, step, outputs -> pinned host, all inside the timed region
    h_in = [t.detach().cpu().pin_memory() for t in (st.x, st.w, st.gy)]
    d_in = [st.x, st.w, st.gy]
    if st.gamma is not None:
        h_in.append(st.gamma.detach().cpu().pin_memory())
        d_in.append(st.gamma)
    d_out = [st.y, st.dx, st.dw]
    h_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in d_out]
    # the step with its copies as one graph: each input is copied on the branch that needs it
    # first, each output leaves as soon as it is final (LayerStep.step_concurrent_host)
    graph_host = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        st.step_concurrent_host(h_in, h_out, stream)
        stream.synchronize()
        with torch.cuda.graph(graph_host, stream=stream):
            st.step_concurrent_host(h_in, h_out, stream)
    e2e_ms = []
    with torch.cuda.stream(stream):
        for i in range(args.warmup + args.steps):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            graph_host.replay()
            e1.record(stream)
            stream.synchronize()
            if i >= args.warmup:
                e2e_ms.append(e0.elapsed_time(e1))
    e2e_serial = max_over_ranks(sum(e2e_ms), "cuda")
    # two steps in flight: a second layer instance (its own device buffers and pinned outputs) and
    # its own graph on a second stream, replayed alternately, so that one step's output copies run
    # beside the next step's input copies (the host link carries both directions at once).  Every
    # step still copies all of its inputs in and all of its outputs out inside the timed region.
    st_b = LayerStep(wl, device=f"cuda:{local_rank}", keep_acc=False, implicit=args.implicit,
                     e4m3_weights=args.e4m3_weights == "on", e4m3_x=args.e4m3_x == "on")
    h_out_b = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in d_out]
    stream_b = torch.cuda.Stream()
    graph_host_b = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream_b):
        st_b.step_concurrent_host(h_in, h_out_b, stream_b)
        stream_b.synchronize()
        with torch.cuda.graph(graph_host_b, stream=stream_b):
            st_b.step_concurrent_host(h_in, h_out_b, stream_b)
    pairs = ((graph_host, stream), (graph_host_b, stream_b))

    def pipelined(k):
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        stream_b.wait_event(e0)
        for i in range(k):
            g, s_ = pairs[i % 2]
            with torch.cuda.stream(s_):
                g.replay()
        done_b = torch.cuda.Event()
        done_b.record(stream_b)
        stream.wait_event(done_b)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    pipelined(max(args.warmup, 4))
    flush.zero_()
    e2e_total = max_over_ranks(pipelined(args.steps), "cuda")
    e2e = {"value": job_tops(ops, args.steps, world, e2e_total), "unit": UNIT,
           "h2d_bytes_per_step": sum(t.numel() * t.element_size() for t in h_in),
           "d2h_bytes_per_step": sum(t.numel() * t.element_size() for t in h_out),
           "timing": "two steps in flight: two layer instances, each step one CUDA graph with its copies "
                     "from and to pinned host memory (each input copied on the branch that needs it first, "
                     "each output as soon as it is final), replayed alternately on two streams so that one "
                     "step's output copies overlap the next step's input copies; one interval over all steps, "
                     "CUDA events; no L2 flush between the steps: every step's inputs arrive from host "
                     "memory over the link during the step",
           "serial": {"value": job_tops(ops, args.steps, world, e2e_serial), "unit": UNIT,
                      "timing": "one step at a time: the same graph replayed after a 256 MiB L2 flush, "
                                "each step timed alone with CUDA events"}}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        r = run_oracle_sample(batch=32, steps=3)
        t = statistics.mean(r["times"][1:])  # the first step runs cold (page faults, caches)
        cpu = {"value": r["ops"] / t / 1e12, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"oracle layer step on 32 of the 128 samples (M={r['M']} K={r['K']} D={r['D']}), "
                         f"mean of 2 runs after one untimed run, {t:.2f} s each, one thread"}
        ncores = host_cores()
        if ncores > 1:
            ra = run_oracle_parallel(batch=32, procs=ncores)
            cpu["all_cores"] = {"value": ra["value"], "unit": UNIT, "cores": ncores, "kind": "oracle",
                                "sample": f"{ncores} single-threaded oracle processes started together after one "
                                          f"untimed step each, each one layer step on its own 32 of the 128 "
                                          f"samples (M={ra['M']} K={ra['K']} D={ra['D']}), {ra['wall_s']:.2f} s "
                                          f"first start to last end"}

    if world > 1:
        dist.barrier()
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "e4m3", "data": "synthetic",
                "config": {"workload": WORKLOAD, "l2": "flushed before every timed step (256 MiB write)",
                           "timing": "CUDA-graph replay of the whole step (three stream branches: pack W | "
                                     "pack X + forward + grad_weight | SCQ + grad_input with the Folder in its "
                                     "epilogue), CUDA events on the launching stream",
                           "parallelism": f"{world} independent replicas" if world > 1 else "1 GPU",
                           "forward": "implicit GEMM (pixel-major sign(X))" if st.implicit
                           else "e4m3 copies of sign(X_u) by TMA (forward and grad_weight)" if st.e4m3_x
                           else "1-bit unfolded X_u",
                           "weights": "e4m3 copies of sign(W) by TMA" if (st.w8 is not None or st.wt8 is not None)
                           else "packed sign(W) expanded per CTA"},
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches_per_step * args.steps,
                "clocks": clocks, "stage_ms": {k: round(v, 5) for k, v in stage_ms.items()}}
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


TABLE5_SHAPES = [(512, 512, 512), (512, 512, 1024), (1024, 512, 512), (1024, 512, 1024), (2048, 512, 512),
                 (2048, 512, 1024)]


def table5(args):
    """Table 5's comparison on this datapath: the product of sign(A) [M, K] and sign(B) [N, K]
    (1-bit, the forward product) against the product of the kept quarter of A's rows as 4-bit
    codes with sign(B) (average 1-bit, b = 4: the grad_input product on a PSQ branch with one
    row per group).  Each product is one graph-captured launch, timed with CUDA events after an
    L2 flush; both write 4-byte outputs (fp32 y, int32 accumulators)."""
    import torch
    from paper_2408_14267_gb300 import build, fqt1
    build.build()
    dev = torch.device("cuda")
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    stream = torch.cuda.Stream()
    gen = torch.Generator(device="cpu").manual_seed(5)

    def timed(fn, reps):
        with torch.cuda.stream(stream):
            fn(stream)
            stream.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fn(stream)
            for _ in range(max(args.warmup, 3)):
                g.replay()
            ts = []
            for _ in range(reps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                g.replay()
                e1.record(stream)
                ts.append((e0, e1))
            stream.synchronize()
        return statistics.median(a.elapsed_time(b) * 1e3 for a, b in ts)

    rows = []
    for M, K, N in TABLE5_SHAPES:
        a = torch.randn(M, K, generator=gen).to(dev)
        b = torch.randn(N, K, generator=gen).to(dev)
        wK = fqt1.packed_words(K)
        sa = torch.empty(M, wK, dtype=torch.int32, device=dev)
        sb_row = torch.empty(N, wK, dtype=torch.int32, device=dev)
        fqt1.binarize_pack(a, M, K, K, sa, None, None)
        fqt1.binarize_pack(b, N, K, K, sb_row, None, None)
        ones = torch.ones(N, device=dev)
        y = torch.empty(M, N, device=dev)
        one_bit = timed(lambda s: fqt1.fwd_gemm(sa, sb_row, M, N, K, ones, None, y, s), args.steps)
        # average 1-bit: the kept quarter of A's rows (b = 4) as 4-bit codes
        g = (torch.randn(M, K, generator=gen) * torch.exp(2 * torch.randn(M, 1, generator=gen))).to(dev)
        p = fqt1.AgpParams(4, 0, 11, 1)
        cap = fqt1.kept_capacity(M, 4, 0)
        q = fqt1.QGradBuffers(M, cap, cap, K, dev)
        ws = fqt1.scq_workspace(M, K, N, 1, dev)
        status = torch.zeros(4, dtype=torch.int32, device=dev)
        fqt1.agp_quantize_grad(g, M, K, 0, None, p, q, ws, status)
        acc = torch.empty(cap, N, dtype=torch.int32, device=dev)
        # contraction over K: the product's second operand is sign(B) packed along K, as for the forward
        avg = timed(lambda s: fqt1.bwd_input_gemm(q, sb_row, None, M, K, N, p, acc, None, s), args.steps)
        rows.append({"M": M, "K": K, "N": N, "kept_rows": q.count(), "one_bit_us": round(one_bit, 2),
                     "avg_1bit_us": round(avg, 2)})
    ratio = statistics.mean(r["avg_1bit_us"] / r["one_bit_us"] for r in rows)
    print(json.dumps({"metric": "GEMM time, average 1-bit (b=4, kept quarter, 4-bit codes) / 1-bit, Table 5 shapes",
                      "value": ratio, "unit": "ratio", "higher_is_better": False, "steps": args.steps,
                      "warmup": args.warmup, "dtype": "e4m3", "data": "synthetic",
                      "config": {"workload": "Table 5 shapes M x K x N, K the contraction",
                                 "l2": "flushed before every timed launch (256 MiB write)",
                                 "timing": "one graph-captured launch, CUDA events, median"},
                      "shapes": rows}))


def layer_sweep(args):
    """The layer step on every VGG-16 (32x32, batch 128) and ResNet-18 (224x224, batch 64) layer
    shape, b = 4 on both SCQ branches: per layer the three-branch step (LayerStep.step_concurrent)
    as one CUDA graph, the L2 flushed before every replay, CUDA events on the launching stream,
    median over `steps` replays.  Reports 6 M K D / time per layer, the fp32 bytes the step reads
    and writes (x, W, gY in; y, dx, dW out) over the same time, each stage's eager device time
    (stage_times), and the whole set's 6 M K D sum over the sum of the layer times."""
    import torch
    from paper_2408_14267_gb300 import build, workloads
    build.build()
    from paper_2408_14267_gb300.layer import LayerStep
    dev = torch.device("cuda")
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)  # 256 MiB > 129 MB L2
    stream = torch.cuda.Stream()
    sets = {"vgg16": lambda: workloads.vgg16_layers(bits=4), "resnet18": workloads.resnet18_imagenet_layers}
    rows = []
    for net in (["vgg16", "resnet18"] if args.layers == "all" else [args.layers]):
        for wl in sets[net]():
            opts = {} if args.colmajor == "auto" else {"colmajor": args.colmajor == "on"}
            st = LayerStep(wl, device=dev, keep_acc=False, e4m3_weights=args.e4m3_weights == "on", **opts)
            with torch.cuda.stream(stream):
                for _ in range(3):
                    st.step()
                stream.synchronize()
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    st.step_concurrent(stream)
                for _ in range(max(args.warmup, 3)):
                    g.replay()
                ts = []
                for _ in range(args.steps):
                    flush.zero_()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                    g.replay()
                    e1.record(stream)
                    ts.append((e0, e1))
                stream.synchronize()
            ms = statistics.median(a.elapsed_time(b) for a, b in ts)
            io = 4 * sum(t.numel() for t in (st.x, st.w, st.gy, st.y, st.dx, st.dw))
            stage_ms = stage_times(st, stream, flush, 5)  # eager, serial: where the step's time goes
            rows.append({"layer": wl["name"], "M": st.M, "K": st.K, "D": st.D, "ms": round(ms, 5),
                         "grad_input": "fused Folder" if st.fold else ("column-major Folder" if st.colmajor
                                                                        else "row-major Folder"),
                         "tops": round(st.dense_ops() / (ms * 1e-3) / 1e12, 2),
                         "fp32_io_gbs": round(io / (ms * 1e-3) / 1e9, 1),
                         "stage_us": {k: round(v * 1e3, 1) for k, v in stage_ms.items()}})
            del g, st
            torch.cuda.empty_cache()
    total_ms = sum(r["ms"] for r in rows)
    total_ops = sum(6.0 * r["M"] * r["K"] * r["D"] for r in rows)
    print(json.dumps({"metric": "effective TOPS of the 1-bit FQT layer step over VGG-16 / ResNet-18 layer shapes",
                      "value": total_ops / (total_ms * 1e-3) / 1e12, "unit": "TOPS", "higher_is_better": True,
                      "steps": args.steps, "warmup": args.warmup, "dtype": "e4m3", "data": "synthetic",
                      "config": {"workload": f"{args.layers} layer shapes, b = 4, keep 1/4, SCQ",
                                 "weights": ("e4m3 copies of sign(W) by TMA" if args.e4m3_weights == "on"
                                             else "packed sign(W) expanded in the products"),
                                 "l2": "flushed before every timed replay (256 MiB write)",
                                 "timing": "one CUDA graph of the three-branch step per layer, CUDA events, median"},
                      "layers": rows}))


SWEEP_SIZES = (1024, 2048, 4096, 8192, 16384)
SWEEP_GROUPS = (64, 128, 256, 512, 1024)
SWEEP_BITS = (1, 2, 4, 8)
SWEEP_ORACLE_MAX = 4096  # the oracle is timed on sweep points up to M = K = D = 4096

SWEEP_ORACLE_SCRIPT = r"""
import json, sys, time
sys.path.insert(0, sys.argv[1])
from paper_2408_14267_gb300 import workloads as wl
from oracle import method as om
M, K, D, G, b, gs = (int(v) for v in sys.argv[2:8])
w = wl.sweep_point(M, K, D, G, b)
rpg = M // G
rows = gs * rpg
x, gy = w["x"][:rows], w["gy"][:rows]
om.layer_step_linear(x[:rpg * b], w["w"], w["gamma"], gy[:rpg * b], b, w["mode_s"], w["seed_s"], b, w["mode_c"],
                     w["seed_c"], rpg)
t0 = time.perf_counter()
om.layer_step_linear(x, w["w"], w["gamma"], gy, b, w["mode_s"], w["seed_s"], b, w["mode_c"], w["seed_c"], rpg)
t = time.perf_counter() - t0
print(json.dumps({"s": t, "ops": 6.0 * rows * K * D, "rows": rows}))
"""


def sweep_points(which):
    if which == "routine":
        return [(4096, 4096, 4096, 256, b) for b in SWEEP_BITS]
    if which == "diag":
        return [(n, n, n, 256, 4) for n in SWEEP_SIZES]
    return [(n, k, n, g, b) for n in SWEEP_SIZES for k in SWEEP_SIZES for g in SWEEP_GROUPS for b in SWEEP_BITS]


def gemm_sweep(args):
    """The throughput sweep over GEMM-shaped linear layers (M = D rows and output channels, K
    input features, `groups` sample groups of M / groups rows, AGP b on both SCQ branches with
    keep ratio 1/b).  Per point one JSON line: the three-branch step as one CUDA graph (L2
    flushed before every replay, CUDA events, mean over `steps` replays), its effective TOPS
    (6 M K D / time), the step's fraction of the fp8 tensor peak (issued product operations
    2 M K D + 2 (kept rows) D K + 2 (kept channels) M K over the time), its fraction of the HBM
    peak counting only the fp32 inputs and outputs (x, W, gY read; y, dx, dW written), each
    product's own tensor fraction from an eager per-stage pass, and, up to 4096, the oracle timed
    on one host core over the first 16 sample groups of the point."""
    import torch
    from paper_2408_14267_gb300 import build, workloads
    build.build()
    from paper_2408_14267_gb300.layer import LayerStep
    dev = torch.device("cuda")
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)  # 256 MiB > 129 MB L2
    stream = torch.cuda.Stream()
    hbm_peak, bf16_peak, peak_src = load_peaks()
    fp8_peak = 2.0 * bf16_peak
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               NUMEXPR_NUM_THREADS="1")
    for (M, K, D, G, b) in sweep_points(args.sweep):
        wl = workloads.sweep_point_device(M, K, D, G, b, dev)
        st = LayerStep(wl, device=dev, keep_acc=False, e4m3_weights=args.e4m3_weights == "on",
                       e4m3_x=args.e4m3_x == "on")
        del wl
        torch.cuda.synchronize()  # the inputs are drawn on the default stream; the step runs on `stream`
        with torch.cuda.stream(stream):
            st.dev_status.zero_()
            for _ in range(3):
                st.step()
            stream.synchronize()
            if int(st.dev_status[0].item()) != 0:
                raise RuntimeError(f"sweep point {(M, K, D, G, b)}: device status {int(st.dev_status[0].item()):#x}")
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                st.step_concurrent(stream)
            for _ in range(max(args.warmup, 3)):
                g.replay()
            ts = []
            for _ in range(args.steps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                g.replay()
                e1.record(stream)
                ts.append((e0, e1))
            stream.synchronize()
        ms = statistics.mean(a.elapsed_time(e) for a, e in ts)
        stage_ms = stage_times(st, stream, flush, 5)
        ks, kc = st.psq.count() * st.rpg, st.pcq.count()
        issued = 2.0 * M * K * D + 2.0 * ks * D * K + 2.0 * kc * M * K
        io = 4.0 * (2 * M * K + 2 * D * K + 2 * M * D)
        sec = ms * 1e-3
        line = {"point": {"M": M, "K": K, "D": D, "groups": G, "bits": b, "kept_rows": ks, "kept_channels": kc},
                "ms": round(ms, 5), "tops": 6.0 * M * K * D / sec / 1e12, "unit": "TOPS",
                "tensor_frac": issued / sec / 1e12 / fp8_peak, "hbm_frac": io / sec / 1e9 / hbm_peak,
                "peaks": {"fp8_tflops": fp8_peak, "hbm_gbs": hbm_peak, "source": peak_src,
                          "note": "fp8 = 2 x bf16 (nominal ratio); HBM fraction counts fp32 I/O only"},
                "gemms": gemm_rooflines(st, stage_ms, bf16_peak, peak_src),
                "stage_ms": {k: round(v, 5) for k, v in stage_ms.items()},
                "config": {"l2": "flushed before every timed replay (256 MiB write)",
                           "x_operand": ("e4m3 copies of sign(X) by TMA" if st.e4m3_x
                                         else "packed sign(X) expanded in the products"),
                           "timing": "one CUDA graph of the three-branch step, CUDA events, mean",
                           "steps": args.steps, "warmup": args.warmup, "data": "synthetic (device draw)"}}
        if max(M, K, D) <= SWEEP_ORACLE_MAX and not args.no_cpu_baseline:
            gs = 16
            p = subprocess.run([sys.executable, "-c", SWEEP_ORACLE_SCRIPT, ROOT, str(M), str(K), str(D), str(G),
                                str(b), str(gs)], env=env, capture_output=True, text=True, timeout=1800)
            if p.returncode == 0:
                r = json.loads(p.stdout.strip().splitlines()[-1])
                line["cpu_baseline"] = {"value": r["ops"] / r["s"] / 1e12, "unit": "TOPS", "cores": 1,
                                        "kind": "oracle",
                                        "sample": f"oracle layer step on the first {gs} of {G} sample groups "
                                                  f"({r['rows']} rows), full K and D, one thread, after one "
                                                  f"untimed step on {b} groups"}
            else:
                line["cpu_baseline"] = {"error": p.stderr[-300:]}
        print(json.dumps(line), flush=True)
        del g, st
        torch.cuda.empty_cache()


def build_model(name, res, binary, classes=10):
    """VGG-16 or ResNet-18 for res x res inputs.  binary: the hidden convolutions and fully
    connected layers are binop layers (1-bit forward, 1-bit FQT backward); the first convolution
    and the classifier stay full precision, as in binary networks; BatchNorm and Hardtanh between
    layers.  Otherwise every layer is a float32 torch layer."""
    import torch
    from paper_2408_14267_gb300 import binop
    nn = torch.nn

    def conv(cin, cout, k, s, p, first=False):
        if binary and not first:
            return binop.Conv2d(cin, cout, k, stride=s, padding=p, qcfg=binop.QuantConfig(4))
        return nn.Conv2d(cin, cout, k, stride=s, padding=p, bias=False)

    def fc(fin, fout, last=False):
        if binary and not last:
            return binop.Linear(fin, fout, qcfg=binop.QuantConfig(4))
        return nn.Linear(fin, fout)

    if name == "vgg16":
        cfg = [64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M", 512, 512, 512, "M"]
        layers, cin = [], 3
        for v in cfg:
            if v == "M":
                layers.append(nn.MaxPool2d(2))
            else:
                layers += [conv(cin, v, 3, 1, 1, first=cin == 3), nn.BatchNorm2d(v), nn.Hardtanh()]
                cin = v
        feat = 512 * (res // 32) ** 2
        layers += [nn.Flatten(), fc(feat, 512), nn.BatchNorm1d(512), nn.Hardtanh(), fc(512, 512),
                   nn.BatchNorm1d(512), nn.Hardtanh(), fc(512, classes, last=True)]
        return nn.Sequential(*layers)

    class Block(nn.Module):
        def __init__(self, cin, cout, stride):
            super().__init__()
            self.c1, self.b1 = conv(cin, cout, 3, stride, 1), nn.BatchNorm2d(cout)
            self.c2, self.b2 = conv(cout, cout, 3, 1, 1), nn.BatchNorm2d(cout)
            self.down = None
            if stride != 1 or cin != cout:
                self.down = nn.Sequential(conv(cin, cout, 1, stride, 0), nn.BatchNorm2d(cout))
            self.act = nn.Hardtanh()

        def forward(self, x):
            y = self.act(self.b1(self.c1(x)))
            y = self.b2(self.c2(y))
            return self.act(y + (x if self.down is None else self.down(x)))

    if res <= 64:  # CIFAR-style stem
        stem = [conv(3, 64, 3, 1, 1, first=True), nn.BatchNorm2d(64), nn.Hardtanh()]
    else:
        stem = [conv(3, 64, 7, 2, 3, first=True), nn.BatchNorm2d(64), nn.Hardtanh(), nn.MaxPool2d(3, 2, 1)]
    blocks, cin = [], 64
    for cout, stride in ((64, 1), (128, 2), (256, 2), (512, 2)):
        blocks += [Block(cin, cout, stride), Block(cout, cout, 1)]
        cin = cout
    return nn.Sequential(*stem, *blocks, nn.AdaptiveAvgPool2d(1), nn.Flatten(), fc(512, classes, last=True))


def model_step(args):
    """One training step (forward, cross-entropy, backward, SGD update) of a synthetic VGG-16 or
    ResNet-18 on random data, graph-captured, with binop layers against float32 torch layers
    (TF32 off): the GPU analogue of Table 3's speedup over FP32 PyTorch."""
    import torch
    from paper_2408_14267_gb300 import build
    build.build()
    torch.backends.cudnn.allow_tf32 = False
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.backends.cudnn.benchmark = True
    dev = torch.device("cuda")
    gen = torch.Generator(device="cpu").manual_seed(1)
    x = torch.randn(args.batch, 3, args.res, args.res, generator=gen).to(dev)
    t = torch.randint(0, 10, (args.batch,), generator=gen).to(dev)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    out = {}
    if args.profile:  # eager steps of the binop model only (for a kernel launch list)
        torch.backends.cudnn.benchmark = False  # no algorithm search among the launches
        torch.manual_seed(2)
        net = build_model(args.model, args.res, True).to(dev)
        opt = torch.optim.SGD(net.parameters(), lr=1e-3)
        for _ in range(args.warmup + args.profile):
            opt.zero_grad(set_to_none=False)
            torch.nn.functional.cross_entropy(net(x), t).backward()
            opt.step()
        torch.cuda.synchronize()
        return
    for arm, binary in (("fp32", False), ("fqt1", True)):
        torch.manual_seed(2)
        net = build_model(args.model, args.res, binary).to(dev)
        opt = torch.optim.SGD(net.parameters(), lr=1e-3)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for _ in range(3):  # warm-up before capture (allocator, cuDNN algorithms)
                opt.zero_grad(set_to_none=False)
                torch.nn.functional.cross_entropy(net(x), t).backward()
                opt.step()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            opt.zero_grad(set_to_none=False)
            loss = torch.nn.functional.cross_entropy(net(x), t)
            loss.backward()
            opt.step()
        for _ in range(max(args.warmup, 3)):
            g.replay()
        ts = []
        for _ in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            g.replay()
            e1.record()
            ts.append((e0, e1))
        torch.cuda.synchronize()
        out[arm] = statistics.median(a.elapsed_time(b) for a, b in ts)
        assert torch.isfinite(loss).item(), "non-finite loss"
    print(json.dumps({"metric": f"training step speedup over FP32 PyTorch, synthetic {args.model}",
                      "value": out["fp32"] / out["fqt1"], "unit": "x", "higher_is_better": True,
                      "steps": args.steps, "warmup": args.warmup, "dtype": "e4m3", "data": "synthetic",
                      "ms_per_step": {"fqt1": round(out["fqt1"], 4), "fp32": round(out["fp32"], 4)},
                      "config": {"workload": f"{args.model}, batch {args.batch}, {args.res}x{args.res} inputs, "
                                             "10 classes; hidden convolutions and fully connected layers binop "
                                             "(1-bit forward, AGP b=4 SCQ backward), first convolution and "
                                             "classifier float32; the fp32 arm has float32 layers (TF32 off)",
                                 "l2": "flushed before every timed step (256 MiB write)",
                                 "timing": "one CUDA graph per arm (forward, loss, backward, SGD step), CUDA "
                                           "events, median; the graph repeats its quantizer seeds"}}))


def variance_study(args):
    """Quantizer variance on heterogeneous synthetic gradients (the mechanism of Sec. 5.2 and the
    quantizer-variance comparison of the experiments): G [M, D] of 128 samples x 64 rows, per-sample
    scales exp(2 N(0,1)), groups = samples.  For each setting, `steps` seeds of the library's AGP
    quantizer (fqt1_agp_quantize_grad) give E||Q(G) - G||^2, summed over elements, next to the bound
    of Eq. 24, D_g / (4 B^2) sum over the N/b largest ranges of R_i^2 (D_g = elements per group),
    and the 1-bit PSQ bound D_g / 4 sum_i R_i^2.  The dequantization Q = S' q + Z' (0 for pruned
    groups) is evaluated here in float64 for the measurement only."""
    import numpy as np
    import torch
    from paper_2408_14267_gb300 import build, fqt1
    build.build()
    dev = torch.device("cuda")
    rng = np.random.default_rng(31)
    N, rpg, D = 128, 64, 256
    M = N * rpg
    g_np = (1e-3 * rng.standard_normal((N, rpg, D)) * np.exp(2 * rng.standard_normal((N, 1, 1)))).reshape(M, D)
    g = torch.from_numpy(g_np.astype(np.float32)).to(dev)
    g64 = g.double()
    ws = fqt1.scq_workspace(M, D, 0, rpg, dev)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    settings = [("PSQ 1-bit", 1, 0), ("AGP b=2", 2, 0), ("AGP b=4", 4, 0), ("AGP b=8", 8, 0),
                ("AGP b=4, Bernoulli masks", 4, 1), ("AGP b=4, top-N/b (biased)", 4, 2)]
    results = []
    for name, bits, mode in settings:
        cap = fqt1.kept_capacity(N, bits, mode)
        q = fqt1.QGradBuffers(N, cap, cap * rpg, D, dev)
        sq = torch.zeros(M, D, dtype=torch.float64, device=dev)
        mean = torch.zeros(M, D, dtype=torch.float64, device=dev)
        for seed in range(args.steps):
            fqt1.agp_quantize_grad(g, M, D, 0, None, fqt1.AgpParams(bits, mode, 1000 + seed, rpg), q, ws, status)
            cnt = q.count()
            kept = q.kept_idx[:cnt].long()
            codes = q.codes[:cnt * rpg, :D].double().view(cnt, rpg, D)
            deq = torch.zeros(N, rpg, D, dtype=torch.float64, device=dev)
            deq[kept] = codes * q.scale[:cnt].double().view(cnt, 1, 1) + q.zero[:cnt].double().view(cnt, 1, 1)
            deq = deq.view(M, D)
            sq += (deq - g64) ** 2
            mean += deq
        assert int(status[0].item()) == 0
        r = q.group_range.double().cpu().numpy()
        B = (1 << bits) - 1
        top = np.sort(r)[::-1][:max(1, N // bits) if bits > 1 else N]
        d_g = rpg * D
        var = float(sq.sum().item()) / args.steps
        bias = float(((mean / args.steps - g64) ** 2).sum().item())
        results.append({"setting": name, "bits": bits, "E_sq_error": var, "sq_bias_of_mean": bias,
                        "eq24_bound": d_g / (4 * B * B) * float(np.sum(top ** 2)),
                        "psq_1bit_bound": d_g / 4 * float(np.sum(r ** 2))})
    agp4 = next(x for x in results if x["setting"] == "AGP b=4")["E_sq_error"]
    psq = results[0]["E_sq_error"]
    print(json.dumps({"metric": "quantizer variance E||Q(G) - G||^2, AGP b=4 / 1-bit PSQ", "value": agp4 / psq,
                      "unit": "ratio", "higher_is_better": False, "steps": args.steps, "data": "synthetic",
                      "config": {"workload": f"G [{M}, {D}]: {N} samples x {rpg} rows, N(0,1) x 1e-3 x exp(2 N(0,1)) "
                                             "per sample; groups = samples; seeds 1000 .. 1000 + steps - 1"},
                      "settings": results}))


def reference_arm(args, world, rank):
    """The reference arm: the oracle, as it stands, timed on the host cores."""
    if rank != 0:
        return
    batch = 32  # a bounded sample of the workload per step (32 of 128 samples)
    r = run_oracle_sample(batch=batch, steps=args.warmup + args.steps)
    times = r["times"][args.warmup:]
    total = sum(times)
    value = r["ops"] * len(times) / total / 1e12
    sample = (f"oracle layer step on {batch} of the 128 samples (M={r['M']} K={r['K']} D={r['D']}) per step, "
              f"one thread")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD}, "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1,
                                                               "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


if __name__ == "__main__":
    main()
