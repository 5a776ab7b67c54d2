"""Benchmark of TRACK's routed denoising hot path on GB300.

Default workload: the Wan-2.1-shaped pair of the paper's Table 1 row (a
14B-shaped large DiT, 5120 wide, 40 blocks, 40 heads, FFN 13824, and a
1.3B-shaped small DiT, 1536 wide, 30 blocks, 12 heads, FFN 8960; bf16, weights
generated on the device), one 480p latent 16x21x60x104 (32760 tokens), text
512x4096, classifier-free guidance 5 (cond and uncond batched: 2 sequences per
forward), 50 flow-matching Euler steps with shift 5, and the top-K policy
(K = 25) of a calibration run over 8 seeds (Sec. 3.2.1, Eq. 4-5), read from the
score map that `bench.py --calibrate` wrote.

One benchmark step is one routed denoise step (Eq. 3): the policy's model
evaluated on the guided pair, with the guidance combine fused into the Euler
update.  The steps walk the routed trajectory in order: the warm-up steps are
its first steps, the timed steps the next ones (a trajectory that ends starts
over from its x_T).  Printed metric: routed denoise steps/s of the timed
steps, plus the full routed and all-large trajectories measured end to end
(latency, speedup, energy), per-class kernel rooflines measured with CUDA
events inside the step, an end-to-end number through the C ABI with host
buffers, clocks sampled during the timed region, and the oracle's CPU
throughput on a bounded sample.

    python bench.py [--steps K] [--warmup W] [--gpus N] [--impl ours|reference]
    python bench.py --calibrate [--workload W]        # writes the score map
    python bench.py --workload mid                    # the mid pair, whole trajectories
    python bench.py --kernel gemm|attention|hbm|forward [--workload W] [--batch B]
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

WORKLOAD = "wan480"
WINDOW_WORKLOADS = ("wan480", "wan720", "serving")   # one denoise step per bench step
METRIC = "routed denoise steps/s"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
SCORE_MAPS = os.path.join(ROOT, "paper_2609_30096_gb300", "score_maps")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "ncu_traffic.json")


def load_peaks():
    try:
        with open(PEAKS_FILE) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return FALLBACK_PEAKS, "fallback"


def source_digest(sources):
    """sha1 over the named files of the package's csrc/ (the kernel's sources)."""
    m = hashlib.sha1()
    for src in sources:
        with open(os.path.join(ROOT, "paper_2609_30096_gb300", "csrc", src), "rb") as f:
            m.update(f.read())
    return m.hexdigest()


def measured_traffic(kernel, workload, work_per_launch):
    """DRAM bytes per launch from the committed ncu record of `kernel` on `workload`,
    scaled to a launch of `work_per_launch` (the record's unit of work); None if the
    kernel's sources changed since the capture or no record exists."""
    try:
        with open(TRAFFIC_FILE) as f:
            rec = json.load(f)[kernel][workload]
        if source_digest(rec["sources"]) != rec["source_sha1"]:
            return None, "kernel changed since the ncu capture"
        per = (rec["dram_read_bytes"] + rec["dram_write_bytes"]) / rec["work"]
        return per * work_per_launch, f"scaled by {rec['work_unit']} from {rec['launch']}"
    except Exception as e:  # noqa: BLE001
        return None, f"no capture ({type(e).__name__})"


def forward_flops(arch, batch):
    """Algorithmic FLOPs of one denoiser evaluation of `batch` sequences (text work excluded)."""
    L, d, F, Lt, l = arch.tokens, arch.dim, arch.ffn, arch.text_len, arch.layers
    per = l * (2 * L * (6 * d * d + 2 * d * F) + 4 * L * L * d + 4 * L * Lt * d) + 4 * L * 64 * d
    return batch * per


def text_flops(arch, batch):
    """Once per request and model: text projection and the blocks' cross-attention K/V."""
    Lt, d, Dt, l = arch.text_len, arch.dim, arch.text_dim, arch.layers
    return batch * (2 * Lt * Dt * d + 2 * Lt * d * d + l * 2 * Lt * d * 2 * d)


def guided_sequences(wl):
    """Sequences per denoiser evaluation: cond (and uncond with guidance) per sample."""
    return wl.batch * (1 if wl.cfg == 1.0 else 2)


def policy_str(pol):
    return "".join("S" if p else "L" for p in pol)


# ---------------------------------------------------------------- calibration score maps
def config_hash(wl):
    """64-bit identifier of everything a score map depends on: the pair's
    architectures and weight seeds, the schedule, the guidance scale and the
    calibration seeds."""
    desc = json.dumps({"large": wl.large.__dict__, "small": wl.small.__dict__,
                       "seeds": [synth.SEED_LARGE, synth.SEED_SMALL, synth.SEED_LATENT,
                                 synth.SEED_COND, synth.SEED_UNCOND],
                       "steps": wl.steps, "shift": wl.shift, "cfg": wl.cfg,
                       "generator": "splitmix64-irwin-hall-4"}, sort_keys=True, default=str)
    return int.from_bytes(hashlib.sha1(desc.encode()).digest()[:8], "little")


def score_map_path(wl):
    return os.path.join(SCORE_MAPS, f"{wl.name}.trkscore")


def load_policy(T, wl):
    """(policy, q, M, provenance) from the committed score map of `wl`."""
    path = score_map_path(wl)
    if not os.path.exists(path):
        raise SystemExit(f"no score map for {wl.name}: run `python bench.py --calibrate "
                         f"--workload {wl.name}` first")
    r, q, h = T.track_score_map_load(path)
    if h != config_hash(wl) or r.shape[1] != wl.steps:
        raise SystemExit(f"{path} was written for another configuration")
    prov = {}
    try:
        with open(path[:-len(".trkscore")] + ".json") as f:
            prov = json.load(f)
    except OSError:
        pass
    return T.track_policy_topk(q, wl.k), q, r.shape[0], prov


def window_steps(n_steps, first, count):
    """Trajectory step index of bench steps first .. first+count-1: the steps walk
    the trajectory in order and start over after its last step."""
    return [(first + s) % n_steps for s in range(count)]


def timed_window(policy, warmup, count):
    """First trajectory step of the timed window: the first start w >= warmup whose
    `count` consecutive steps (walked as window_steps) split between the models
    as the whole policy does (count * K / N small steps, rounded), so that the
    timed steps' rate is that of the routed trajectory; failing an exact split,
    the closest one."""
    n = len(policy)
    target = round(count * int(np.sum(policy)) / n)
    best, best_err = warmup, None
    for w in range(warmup, warmup + n):
        err = abs(sum(int(policy[i]) for i in window_steps(n, w, count)) - target)
        if best_err is None or err < best_err:
            best, best_err = w, err
        if err == 0:
            break
    return best


# ---------------------------------------------------------------- ranks (replicas)
def rank_env():
    """(rank, local_rank, world) from the torchrun environment (1 process if absent)."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def rank_first_sample(rank, batch):
    """First evaluation sample of a rank: ranks serve disjoint requests (weak scaling)."""
    return rank * batch


def max_over_ranks(ms, world, device=None):
    """Slowest rank's time (the job's time); a barrier brackets the reduction."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as tdist
    t = torch.tensor([float(ms)], device=device)
    tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    tdist.barrier()
    return float(t.item())


def job_throughput(world, steps_per_trajectory, batch, trajectories, ms):
    """Routed denoise steps per second of the whole job: every rank ran `trajectories`."""
    return world * steps_per_trajectory * batch * trajectories / (ms / 1e3)


def gpu_uuid(index):
    """NVML/nvidia-smi identifier of CUDA device `index` ("GPU-<uuid>"), or None."""
    try:
        import torch
        return "GPU-" + str(torch.cuda.get_device_properties(index).uuid)
    except Exception:  # noqa: BLE001
        return None


class EnergyMeter:
    """Reads the GPU's total-energy counter (NVML, millijoules since driver load)."""

    def __init__(self, index):
        import ctypes
        self.h = None
        try:
            self.lib = ctypes.CDLL("libnvidia-ml.so.1")
            if self.lib.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            uuid = gpu_uuid(index)
            rc = (self.lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) if uuid
                  else self.lib.nvmlDeviceGetHandleByIndex_v2(index, ctypes.byref(h)))
            if rc == 0:
                self.h = h
        except OSError:
            pass

    def read_mj(self):
        import ctypes
        if self.h is None:
            return None
        v = ctypes.c_ulonglong()
        if self.lib.nvmlDeviceGetTotalEnergyConsumption(self.h, ctypes.byref(v)) != 0:
            return None
        return int(v.value)


class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", gpu_uuid(self.index) or str(self.index),
                 f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 8 and parts[0].replace(".", "").isdigit():
                    rows.append(parts)
        except Exception:
            pass
        finally:
            try:
                os.unlink(self.path)
            except Exception:
                pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [float(r[0]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower() == "active"})
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(rows[0][1]),
                "power_w_max": max(float(r[2]) for r in rows if r[2].replace(".", "").isdigit()),
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------- CPU oracle sample
def block_flops(arch, tokens):
    """Algorithmic FLOPs of one transformer block over `tokens` tokens of one sequence."""
    d, F, Lt = arch.dim, arch.ffn, arch.text_len
    return 2 * tokens * (6 * d * d + 2 * d * F) + 4 * tokens * tokens * d + 4 * tokens * Lt * d


class OracleSample:
    """The oracle on a bounded sample of the workload: one DiT block of each model
    (fp64 numpy) over the first `frames` latent frames of the workload's latent
    (all of them when frames is None), or over the first `rows` token rows of
    its first frame, timed and extrapolated to one full-size forward of one
    sequence by algorithmic FLOPs (block FLOPs at the full token count over
    those at the sample's) times the model's depth."""

    def __init__(self, wl, frames=None, rows=None):
        from oracle import dit

        self.wl = wl
        rng = np.random.default_rng(0)
        self.parts = {}
        for which, arch, seed in (("large", wl.large, synth.SEED_LARGE),
                                  ("small", wl.small, synth.SEED_SMALL)):
            f = arch.frames if frames is None else min(frames, arch.frames)
            if rows is not None:
                f = 1
            hgt = arch.height if rows is None else min(arch.height, 2 * rows)
            sample = synth.Arch(**{**arch.__dict__, "layers": 1, "frames": f, "height": hgt})
            specs = [s for s in synth.weight_specs(arch)
                     if not s.name.startswith("blk") or s.name.startswith("blk0.")]
            w = {s.name: synth.make_tensor(s, seed) for s in specs}
            m = dit.DiT(sample, w, "bf16")
            x = rng.normal(size=(sample.tokens, arch.dim))
            _, e0 = m.time_embedding(np.float32(500.0))
            c = m.text_projection(synth.draw(1, 0, (arch.text_len, arch.text_dim), 1.0))
            scale = block_flops(arch, arch.tokens) / block_flops(arch, sample.tokens)
            self.parts[which] = (m, x, e0, c, arch.layers * scale)
        tok = self.parts["large"][0].arch.tokens
        self.description = (
            f"one DiT block of each model (oracle, fp64 numpy) over {tok} of the "
            f"{wl.large.tokens} tokens, extrapolated by block FLOPs to the full latent and "
            f"x layers x sequences per evaluation ({guided_sequences(wl)}); embedding, head "
            f"and text work not included")

    def forward_seconds(self):
        """Extrapolated seconds of one full-size forward of one sequence, per model."""
        t = {}
        for which, (m, x, e0, c, factor) in self.parts.items():
            t0 = time.perf_counter()
            m.block(0, x, e0, c)
            t[which] = (time.perf_counter() - t0) * factor
        return t

    def step_seconds(self, n_large, n_small):
        """Extrapolated seconds per denoise step over a mix of large and small steps."""
        t = self.forward_seconds()
        n = n_large + n_small
        return guided_sequences(self.wl) * (n_large * t["large"] + n_small * t["small"]) / n


def cpu_cores():
    """(threads the oracle's BLAS uses, os.cpu_count())."""
    n = None
    try:
        from threadpoolctl import threadpool_info
        b = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if b:
            n = int(max(b))
    except Exception:
        pass
    return (n or os.cpu_count()), os.cpu_count()


def read_score_map(path):
    """(r [M, N], q [N], config_hash) of a score-map file, parsed on the host (the
    little-endian layout of track_score_map_save)."""
    with open(path, "rb") as f:
        b = f.read()
    if b[:8] != b"TRKSCORE" or int.from_bytes(b[8:12], "little") != 1:
        raise SystemExit(f"{path}: not a score map")
    M, N = int.from_bytes(b[12:16], "little"), int.from_bytes(b[16:20], "little")
    h = int.from_bytes(b[20:28], "little")
    v = np.frombuffer(b[28:28 + 4 * (M * N + N)], dtype="<f4")
    return v[:M * N].reshape(M, N).copy(), v[M * N:].copy(), h


# ---------------------------------------------------------------- reference arm
def run_reference(args):
    """The oracle, as it stands, on the host cores: each bench step times a bounded
    sample of the same workload and converts it to the metric's unit."""
    from oracle import track as otrack

    rank, _, _ = rank_env()
    if rank != 0:
        return 0  # the oracle baseline runs once, on rank 0
    wl = synth.WORKLOADS[args.workload]
    if wl.name in WINDOW_WORKLOADS:
        _, q, h = read_score_map(score_map_path(wl))
        if h != config_hash(wl):
            raise SystemExit("score map written for another configuration")
        pol = otrack.topk_policy(q, wl.k)
        idx = window_steps(wl.steps, timed_window(pol, args.warmup, args.steps), args.steps)
        n_small = int(sum(int(pol[i]) for i in idx))
        mix = (args.steps - n_small, n_small)
        # warm-up + timed steps each run a sample: 8 token rows of the first frame
        # (416 tokens at 480p) keep the whole run to a few minutes on the host
        sampler = OracleSample(wl, rows=8)
    else:
        pol = None
        n_small = wl.k
        mix = (wl.steps - wl.k, wl.k)
        sampler = OracleSample(wl)
    for _ in range(args.warmup):
        sampler.step_seconds(*mix)
    times = [sampler.step_seconds(*mix) for _ in range(args.steps)]
    sec = float(np.mean(times))
    value = wl.batch / sec
    threads, ncpu = cpu_cores()
    cpu = {"value": value, "unit": "steps/s", "cores": threads, "host_cpus": ncpu,
           "kind": "oracle", "sample": sampler.description}
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": sec * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.description, "global_batch": wl.batch,
                   "seq_len": wl.large.tokens,
                   "steps_large_small": list(mix)},
        "cpu_baseline": cpu,
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------- calibration command
def setup_library(args):
    """Builds and loads the library and applies the schedule flags."""
    import paper_2609_30096_gb300 as T
    from paper_2609_30096_gb300 import _build

    _build.build()
    T.track_gemm_schedule(GEMM_SCHEDULES[args.gemm_schedule])
    T.track_gemm_raster(args.gemm_raster)
    T.track_attention_schedule(GEMM_SCHEDULES[args.attn_schedule]
                               | (T.ATTN_ONE_TILE if args.attn_one_tile else 0))
    return T


def run_calibrate(args):
    """Calibration of Sec. 3.2.1 (Eq. 4-5) for the workload on its calibration
    seeds, written to the package's score map of that workload.  Samples are
    calibrated `--calib-batch` at a time and the map is saved after every batch,
    so an interrupted run resumes from the rows already saved."""
    import torch

    wl = synth.WORKLOADS[args.workload]
    torch.cuda.set_device(0)
    T = setup_library(args)
    M = args.seeds or wl.calib_seeds
    batch = args.calib_batch or (2 if wl.large.dim >= 5120 else M)
    sig = T.track_schedule(wl.steps, wl.shift)
    L = T.track_model_create_seeded(wl.large, synth.SEED_LARGE, T.BF16)
    S = T.track_model_create_seeded(wl.small, synth.SEED_SMALL, T.BF16)
    uses_uncond = wl.cfg != 1.0
    path = score_map_path(wl)
    meta_path = path[:-len(".trkscore")] + ".json"
    os.makedirs(SCORE_MAPS, exist_ok=True)
    rows, meta = [], {"workload": wl.description, "config_hash": f"{config_hash(wl):016x}",
                      "seeds": f"calibration samples 0..{M - 1} (latent {synth.SEED_LATENT}+j, "
                               f"cond {synth.SEED_COND}+j, uncond {synth.SEED_UNCOND}+j)",
                      "batches": []}
    if os.path.exists(path) and not args.fresh:
        r0, _, h = T.track_score_map_load(path)
        if h == config_hash(wl) and r0.shape[1] == wl.steps:
            rows = list(r0[:M])
            try:
                with open(meta_path) as f:
                    meta["batches"] = json.load(f).get("batches", [])
            except OSError:
                pass
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    while len(rows) < M:
        first = len(rows)
        b = min(batch, M - first)
        x, c, u = synth.calibration_inputs(wl.large, first, b, uses_uncond)
        xd, cd = torch.from_numpy(x).cuda(), torch.from_numpy(c).cuda()
        ud = torch.from_numpy(u).cuda() if uses_uncond else None
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        r = T.track_calibrate(L, S, xd, cd, ud, wl.cfg, sig, stream=stream.cuda_stream)
        ev1.record(stream)
        T.track_sync(stream.cuda_stream)
        rows.extend(r.cpu().numpy().T)
        meta["batches"].append({"samples": [first, first + b], "seconds": ev0.elapsed_time(ev1) / 1e3})
        meta["M"] = len(rows)
        T.track_score_map_save(path, np.stack(rows), config_hash(wl))
        with open(meta_path, "w") as f:
            json.dump(meta, f, indent=1)
        print(json.dumps({"calibrated": [first, first + b], "of": M,
                          "seconds": meta["batches"][-1]["seconds"]}), flush=True)
        del xd, cd, ud, r
    _, q, _ = T.track_score_map_load(path)
    print(json.dumps({"score_map": path, "q": [float(v) for v in q],
                      "policy": policy_str(T.track_policy_topk(q, wl.k))}))
    return 0


# ---------------------------------------------------------------- the default: routed steps
def class_summary(prof, peaks):
    """Per-class kernel time and rate from track_profile_read's sums."""
    out = {}
    for k, (ms, work, n) in prof.items():
        if not n:
            continue
        rec = {"ms": ms, "launches": int(n), "avg_launch_ms": ms / n}
        if k in ("gemm", "attention", "cross_attention"):
            rec["tflops"] = work / (ms / 1e3) / 1e12 if ms else None
            rec["frac_of_sustained"] = rec["tflops"] / peaks["bf16_tflops_sustained"] if ms else None
        else:
            rec["gb_per_s"] = work / (ms / 1e3) / 1e9 if ms else None
            rec["frac_of_hbm"] = rec["gb_per_s"] / peaks["hbm_gbs"] if ms else None
            rec["bytes_per_launch"] = work / n
        out[k] = rec
    return out


# class of track_profile_read -> the graph-timed entry of the same kernel
GRAPH_TIMED = {"update": "cfg_euler", "disagreement": "disagreement_update"}


def annotate_event_timed(classes, hbm):
    """Beside the per-launch event timing of the microsecond-scale update and Eq. 4
    kernels (whose event pairs cost about as much as the kernel), the rate of the
    same kernel recorded back to back in a CUDA graph at the workload's size.
    Calibration's Eq. 4 is the one fused with its update."""
    for cls, key in GRAPH_TIMED.items():
        if cls in classes and key in hbm:
            classes[cls]["graph_timed_frac_of_hbm"] = hbm[key]["frac_of_hbm"]
            classes[cls]["graph_timed_gb_per_s"] = hbm[key]["gb_per_s"]
            classes[cls]["note"] = ("one CUDA event pair around each microsecond-scale launch; "
                                    "graph_timed_* is the same kernel back to back in a CUDA "
                                    f"graph (hbm_kernels.{key})")
    return classes


def run_window(args):
    """Routed denoise steps of a 14B/1.3B workload (module docstring)."""
    import torch
    import torch.distributed as tdist

    rank, local, world = rank_env()
    torch.cuda.set_device(local)
    if world > 1:
        tdist.init_process_group("nccl")
    T = setup_library(args)
    wl = synth.WORKLOADS[args.workload]
    B, w, N = wl.batch, wl.cfg, wl.steps
    uses_uncond = w != 1.0
    nseq = guided_sequences(wl)
    sig = T.track_schedule(N, wl.shift)
    L = T.track_model_create_seeded(wl.large, synth.SEED_LARGE, T.BF16)
    S = T.track_model_create_seeded(wl.small, synth.SEED_SMALL, T.BF16)
    policy, q, M, prov = load_policy(T, wl)
    all_l = np.zeros(N, np.uint8)

    dev = torch.device("cuda", local)
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.set_stream(stream)
    sid = stream.cuda_stream
    x0, c0, u0 = synth.evaluation_inputs(wl.large, rank_first_sample(rank, B), B, uses_uncond)
    xh = torch.from_numpy(x0).pin_memory()            # x_T of this rank's request(s)
    ch = torch.from_numpy(c0).pin_memory()
    uh = torch.from_numpy(u0).pin_memory() if uses_uncond else None
    x_init = xh.to(dev)
    xd = x_init.clone()
    cd = ch.to(dev)
    ud = uh.to(dev) if uses_uncond else None
    x_host = torch.empty_like(xh).pin_memory()         # the host-driven loop's latent

    def event():
        return torch.cuda.Event(enable_timing=True)

    def step(i, pol, x):
        if i == 0:
            x.copy_(x_init)                            # a trajectory starts from x_T
        T.track_sample(L, S, pol[i:i + 1], sig[i:i + 2], x, cd, ud, w, stream=sid)

    def step_e2e(i, pol):
        # The latent lives on the host between steps: copy it and the request's
        # conditioning in, run the step, read the new latent back.
        xd.copy_(xh if i == 0 else x_host, non_blocking=True)
        cd.copy_(ch, non_blocking=True)
        if uses_uncond:
            ud.copy_(uh, non_blocking=True)
        T.track_sample(L, S, pol[i:i + 1], sig[i:i + 2], xd, cd, ud, w, stream=sid)
        x_host.copy_(xd, non_blocking=True)

    def run(indices, fn):
        """Runs the steps back to back, bracketed by a barrier and a device sync on both
        sides, with an event between steps: (total ms over ranks, per-step ms, launches)."""
        if world > 1:
            tdist.barrier()
        torch.cuda.synchronize()
        n0 = T.track_launch_count()
        marks = [event() for _ in range(len(indices) + 1)]
        marks[0].record(stream)
        for s, i in enumerate(indices):
            fn(i)
            marks[s + 1].record(stream)
        torch.cuda.synchronize()
        T.track_sync(sid)
        per = [marks[s].elapsed_time(marks[s + 1]) for s in range(len(indices))]
        total = marks[0].elapsed_time(marks[-1])
        return max_over_ranks(total, world, dev), per, T.track_launch_count() - n0

    # The timed steps are the window of the routed trajectory that timed_window
    # picks; the latent is first advanced to W steps before it (untimed set-up),
    # then the W warm-up steps run, then the timed ones.
    w0 = timed_window(policy, args.warmup, args.steps)
    for i in window_steps(N, 0, w0 - args.warmup):
        step(i, policy, xd)
    for i in window_steps(N, w0 - args.warmup, args.warmup):
        step(i, policy, xd)
    torch.cuda.synchronize()
    x_at_window = xd.clone()
    idx = window_steps(N, w0, args.steps)
    n_small = int(sum(int(policy[i]) for i in idx))
    n_large = args.steps - n_small

    energy = EnergyMeter(local)
    with ClockSampler(local) as clk:
        ms, per_step, launches = run(idx, lambda i: step(i, policy, xd))
    clocks = clk.summary()
    value = world * B * args.steps / (ms / 1e3)
    fl = n_large * forward_flops(wl.large, nseq) + n_small * forward_flops(wl.small, nseq)
    tflops = fl / (ms / 1e3) / 1e12

    # kernel classes: the window's first steps again, every launch bracketed by events
    peaks, src = load_peaks()
    xp = x_at_window.clone()
    T.track_profile_read()
    T.track_profile_enable(True)
    try:
        n_prof = min(args.steps, args.profile_steps)
        run(idx[:n_prof], lambda i: step(i, policy, xp))
        prof = T.track_profile_read()
        # one calibration step (Sec. 3.2.1: both models on the same latent, Eq. 4, the
        # large model's update) at the middle of the schedule, for its cost and Eq. 4's rate
        k = N // 2
        xc = x_at_window.clone()
        ca, cb = event(), event()
        ca.record(stream)
        T.track_calibrate(L, S, xc, cd, ud, w, sig[k:k + 2], stream=sid)
        cb.record(stream)
        T.track_sync(sid)
        calib_step_ms = ca.elapsed_time(cb)
        prof_calib = T.track_profile_read()
    finally:
        T.track_profile_enable(False)
    del xp, xc
    classes = class_summary(prof, peaks)
    if "disagreement" in class_summary(prof_calib, peaks):
        classes["disagreement"] = class_summary(prof_calib, peaks)["disagreement"]
    dominant = max(("gemm", "attention"), key=lambda c: classes.get(c, {}).get("ms", 0.0))
    dm, dwork, dn = prof[dominant]
    kname = "k_gemm_tc" if dominant == "gemm" else "k_attn_pp (self-attention)"
    achieved = dwork / (dm / 1e3) / 1e12
    peak = peaks["bf16_tflops_sustained"]
    traffic, traffic_src = measured_traffic(kname.split()[0], wl.name, dwork / dn)
    roof = {"bound": "tensor", "kernel": kname, "achieved": achieved, "peak": peak,
            "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
            "peak_source": f"{src} bf16 sustained (a step lasts seconds under the power cap; "
                           f"burst {peaks['bf16_tflops']})",
            "frac_of_burst": achieved / peaks["bf16_tflops"],
            "traffic_unit": "bytes per launch", "traffic_source": traffic_src,
            "launches": int(dn), "avg_launch_ms": dm / dn,
            "share_of_timed_kernels": dm / sum(v[0] for v in prof.values()),
            "measured_in": f"the first {n_prof} timed steps run again with a CUDA event "
                           "before and after every kernel of the classes below"}

    # the update and Eq. 4 kernels at this workload's size, graph-timed (a call lasts
    # microseconds: a CUDA event pair around one call would mostly time the launch)
    hbm = workload_hbm_kernels(T, torch, stream, B, wl.large.latent_numel, peaks)
    annotate_event_timed(classes, hbm)

    # e2e: the same steps through the C ABI with the latent on the host between steps
    x_host.copy_(x_at_window)
    ms_e2e, _, _ = run(idx, lambda i: step_e2e(i, policy))
    e2e_value = world * B * args.steps / (ms_e2e / 1e3)

    # without the whole trajectories: the same number of steps of the all-large
    # trajectory from the window's first step, for the routed / all-large ratio
    all_large_window = None
    if args.no_trajectories:
        xa = x_at_window.clone()
        ms_al, _, _ = run(idx, lambda i: step(i, all_l, xa))
        del xa
        all_large_window = {"steps_per_s": world * B * args.steps / (ms_al / 1e3),
                            "ms_per_step": ms_al / args.steps,
                            "routed_speedup": ms_al / ms,
                            "note": "the timed window's steps run with the large model only"}

    # whole trajectories, end to end (text projection included): routed and all-large
    traj = {}
    if not args.no_trajectories:
        for name, pol in (("routed", policy), ("all_large", all_l)):
            T.track_invalidate_ctx(L)
            T.track_invalidate_ctx(S)
            e0 = energy.read_mj()
            t_ms, per, _ = run(list(range(N)), lambda i, pol=pol: step(i, pol, xd))
            e1 = energy.read_mj()
            traj[name] = {"s": t_ms / 1e3, "per_step_ms": per,
                          "joules": (e1 - e0) / 1e3 if None not in (e0, e1) else None}
        cl = float(np.mean(traj["all_large"]["per_step_ms"][1:]))
        cs = float(np.mean([t for t, p in zip(traj["routed"]["per_step_ms"], policy) if p])) \
            if policy.any() else None
        model_s = ((N - wl.k) * cl + wl.k * (cs or 0.0)) / 1e3
        for name in traj:
            traj[name].pop("per_step_ms")
        ja, jr = traj["all_large"]["joules"], traj["routed"]["joules"]
        traj.update({
            "routed_steps_per_s": world * B * N / traj["routed"]["s"],
            "speedup": traj["all_large"]["s"] / traj["routed"]["s"],
            "ideal_flop_speedup": N / ((N - wl.k) + wl.k * forward_flops(wl.small, 1)
                                       / forward_flops(wl.large, 1)),
            "C_large_ms": cl, "C_small_ms": cs,
            "cost_model": {"routed_s": model_s,
                           "rel_err": abs(model_s - traj["routed"]["s"]) / traj["routed"]["s"],
                           "note": "Eq. 3 cost model: (N - K) C_L + K C_S from the measured "
                                   "per-step costs against the measured routed trajectory"},
            "energy_savings": (1.0 - jr / ja) if ja and jr else None})

    cpu = None
    if rank == 0 and not args.skip_cpu:
        sampler = OracleSample(wl, frames=1)
        sec = sampler.step_seconds(n_large, n_small)
        threads, ncpu = cpu_cores()
        cpu = {"value": B / sec, "unit": "steps/s", "cores": threads, "host_cpus": ncpu,
               "kind": "oracle", "sample": sampler.description}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": wl.description, "global_batch": world * B,
                       "seq_len": wl.large.tokens, "sequences_per_forward": nseq,
                       "parallelism": f"replicas x{world}",
                       "timed_steps": f"trajectory steps {idx[0]}..{idx[-1]} of the {N}-step "
                                      f"routed trajectory, the first window of {args.steps} steps "
                                      f"from step {args.warmup} with the policy's large/small "
                                      f"split (warm-up: the {args.warmup} steps before it)",
                       "steps_large_small": [n_large, n_small],
                       "policy": policy_str(policy),
                       "l2": "inputs larger than L2: every large step streams the 28.6 GB of "
                             "bf16 weights and GB-sized activations through the 126 MB L2",
                       "launch": "eager, one track_sample call per step"},
            "dit_tflops": tflops, "dit_frac_of_sustained": tflops / peaks["bf16_tflops_sustained"],
            "trajectory": traj or None,
            "all_large_window": all_large_window,
            "calibration": {"score_map": os.path.relpath(score_map_path(wl), ROOT), "seeds": M,
                            "seconds": sum(b["seconds"] for b in prov.get("batches", [])) or None,
                            "q": [float(v) for v in q], "step_ms": calib_step_ms},
            "kernels": classes,
            "hbm_kernels": hbm,
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "steps/s",
                    "h2d_bytes_per_step": int(xh.numel() * 4 + ch.numel() * 4 +
                                              (uh.numel() * 4 if uses_uncond else 0)),
                    "d2h_bytes_per_step": int(xh.numel() * 4)},
            "gpu_launches": int(launches),
            "clocks": clocks,
        }
        print(json.dumps(line))
    L.close()
    S.close()
    if world > 1:
        tdist.destroy_process_group()
    return 0
# ---------------------------------------------------------------- whole trajectories (tiny, mid)
def run_trajectories(args):
    """Whole routed trajectories of a small workload (tiny, mid): each timed unit is
    one trajectory of the request (text projection, the policy's N denoiser
    evaluations, fused guidance + Euler updates) replayed from a CUDA graph;
    `--steps` counts trajectories here and the line reports per denoise step.
    The policy comes from a calibration run on the workload's seeds, executed and
    timed before the timed region."""
    import torch
    import torch.distributed as tdist

    rank, local, world = rank_env()
    torch.cuda.set_device(local)
    if world > 1:
        tdist.init_process_group("nccl")
    T = setup_library(args)

    wl = synth.WORKLOADS[args.workload]
    B = wl.batch
    w = wl.cfg
    sig = T.track_schedule(wl.steps, wl.shift)
    L = T.track_model_create_seeded(wl.large, synth.SEED_LARGE, T.BF16)
    S = T.track_model_create_seeded(wl.small, synth.SEED_SMALL, T.BF16)
    uses_uncond = w != 1.0

    # --- offline calibration on wl.calib_seeds seeds (batched), untimed in the step
    xc, cc, uc = synth.calibration_inputs(wl.large, 0, wl.calib_seeds, uses_uncond)
    dev = torch.device("cuda", local)
    xcd = torch.from_numpy(xc).to(dev)
    ccd = torch.from_numpy(cc).to(dev)
    ucd = torch.from_numpy(uc).to(dev) if uses_uncond else None
    # All device work runs on one created stream: CUDA graphs cannot be recorded on the
    # legacy default stream.
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.set_stream(stream)
    sid = stream.cuda_stream
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    r = T.track_calibrate(L, S, xcd, ccd, ucd, w, sig, stream=sid)
    ev1.record(stream)
    T.track_sync()
    calib_ms = ev0.elapsed_time(ev1)
    q = T.track_mean_score(r.cpu().numpy().T)
    policy = T.track_policy_topk(q, wl.k)
    del xcd, ccd, ucd, r

    # --- request inputs: per-rank disjoint evaluation seeds
    x0, c0, u0 = synth.evaluation_inputs(wl.large, rank_first_sample(rank, B), B, uses_uncond)
    xh = torch.from_numpy(x0).pin_memory()
    ch = torch.from_numpy(c0).pin_memory()
    uh = torch.from_numpy(u0).pin_memory() if uses_uncond else None
    xd = torch.empty_like(xh, device=dev)
    cd = ch.to(dev)
    ud = uh.to(dev) if uses_uncond else None
    out_h = torch.empty_like(xh).pin_memory()

    x_init = xh.to(dev)

    # One trajectory (text projection included) replayed from a CUDA graph recorded
    # per policy; step_eager is the same work launched kernel by kernel (the fallback of
    # the event-bracketed kernel timing).
    def step_device(pol):
        xd.copy_(x_init)                          # on-device reset of the latent
        T.track_sample_graph(L, S, pol, sig, xd, cd, ud, w, stream=sid)

    def step_eager(pol):
        xd.copy_(x_init)
        T.track_invalidate_ctx(L)
        T.track_invalidate_ctx(S)
        T.track_sample(L, S, pol, sig, xd, cd, ud, w, stream=sid)

    def step_e2e(pol):
        xd.copy_(xh, non_blocking=True)           # host -> device: latent and text
        cd.copy_(ch, non_blocking=True)
        if uses_uncond:
            ud.copy_(uh, non_blocking=True)
        T.track_sample_graph(L, S, pol, sig, xd, cd, ud, w, stream=sid)
        out_h.copy_(xd, non_blocking=True)        # device -> host: the sample

    def prime(pol):                               # eager run, then the graph's recording
        step_device(pol)
        step_device(pol)

    def timed(fn, pol, steps):
        if world > 1:
            tdist.barrier()
        torch.cuda.synchronize()
        n0 = T.track_launch_count()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(steps):
            fn(pol)
        b.record(stream)
        torch.cuda.synchronize()
        T.track_sync(sid)
        ms = a.elapsed_time(b)
        launches = T.track_launch_count() - n0
        return max_over_ranks(ms, world, dev), launches

    def profiled_pass(pol, steps):
        # Replays a copy of the trajectory's graph recorded with timing on (an event-
        # record node before and after each bracketed kernel), reading the brackets after
        # every replay.  Falls back to kernel-by-kernel launches if that fails.
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def bracketed(fn):
            tot = {k: [0.0, 0.0, 0] for k in T.PROFILE_CLASSES}
            ms_tot = 0.0
            torch.cuda.synchronize()
            T.track_profile_read()                    # drop the priming calls' records
            for _ in range(steps):
                a.record(stream)
                fn(pol)
                b.record(stream)
                torch.cuda.synchronize()
                ms_tot += a.elapsed_time(b)
                for k, v in T.track_profile_read().items():
                    tot[k] = [x + y for x, y in zip(tot[k], v)]
            return ms_tot, tot

        T.track_profile_enable(True)
        try:
            try:
                prime(pol)                            # eager run, then the bracketed recording
                mode = "graph"
                ms_tot, tot = bracketed(step_device)
            except T.TrackError:
                mode = "eager"
                ms_tot, tot = bracketed(step_eager)
        finally:
            T.track_profile_enable(False)
        return max_over_ranks(ms_tot, world, dev), {k: tuple(v) for k, v in tot.items()}, mode

    for _ in range(args.warmup):                   # the first two record the graph
        step_device(policy)
    for _ in range(2):
        step_eager(policy)
    torch.cuda.synchronize()
    T.track_profile_read()                         # drop any stale records

    energy = EnergyMeter(local)
    with ClockSampler(local) as clk:
        e0 = energy.read_mj()
        ms, launches = timed(step_device, policy, args.steps)
        e1 = energy.read_mj()
    clocks = clk.summary()
    # Same steps again with every GEMM / attention / norm launch bracketed by CUDA events
    # on its stream (the brackets cost a few percent, so `value` comes from the pass above).
    ms_prof, prof, prof_mode = profiled_pass(policy, args.steps)

    all_l = np.zeros(wl.steps, np.uint8)
    prime(all_l)
    for _ in range(max(1, args.warmup // 2)):
        step_device(all_l)
    e2 = energy.read_mj()
    ms_all_large, _ = timed(step_device, all_l, args.steps)
    e3 = energy.read_mj()
    joules = None
    if None not in (e0, e1, e2, e3):
        jr, ja = (e1 - e0) / 1e3 / args.steps, (e3 - e2) / 1e3 / args.steps
        joules = {"routed_j_per_trajectory": jr, "all_large_j_per_trajectory": ja,
                  "savings": 1.0 - jr / ja if ja > 0 else None,
                  "source": "NVML total energy counter around the timed passes"}

    # Cost model of Eq. 3 (total ~ sum_i C_pi(i)): latency against the switching budget K,
    # and the equal-budget policies of the paper's ablation at the workload's K.
    nsw = max(3, args.steps // 2)
    sweep = []
    for kk in range(wl.steps + 1):
        pol = T.track_policy_topk(q, kk)
        prime(pol)
        t, _ = timed(step_device, pol, nsw)
        sweep.append({"K": kk, "ms": t / nsw, "policy": "".join("S" if p else "L" for p in pol)})
    c_l, c_s = sweep[0]["ms"] / wl.steps, sweep[-1]["ms"] / wl.steps
    cost_err = max(abs(r["ms"] - ((wl.steps - r["K"]) * c_l + r["K"] * c_s)) / r["ms"] for r in sweep)
    equal_budget = {}
    for name, pol in (("top_k", policy), ("first_k", T.track_policy_first_k(wl.steps, wl.k)),
                      ("last_k", T.track_policy_last_k(wl.steps, wl.k)),
                      ("random_k", T.track_policy_random_k(wl.steps, wl.k, synth.SEED_EVAL))):
        prime(pol)
        t, _ = timed(step_device, pol, nsw)
        equal_budget[name] = {"ms": t / nsw, "policy": "".join("S" if p else "L" for p in pol)}
    # The same routed and all-large trajectories over the history-carrying
    # multistep scheduler (Eq. 2 with h_i), launched kernel by kernel.
    ms_state = torch.empty(2 * xd.numel(), dtype=torch.float32, device=dev)

    def step_multistep(pol):
        xd.copy_(x_init)
        T.track_invalidate_ctx(L)
        T.track_invalidate_ctx(S)
        T.track_sample_multistep(L, S, pol, sig, xd, cd, ud, w, state=ms_state, stream=sid)

    multistep = {}
    for name, pol in (("routed", policy), ("all_large", all_l)):
        step_multistep(pol)
        t, _ = timed(step_multistep, pol, nsw)
        multistep[name + "_ms"] = t / nsw
    multistep["speedup"] = multistep["all_large_ms"] / multistep["routed_ms"]
    multistep["scheduler"] = "second-order predictor-corrector with history (Eq. 2 h_i)"

    for _ in range(max(1, args.warmup // 2)):
        step_e2e(policy)
    ms_e2e, _ = timed(step_e2e, policy, args.steps)

    per_traj_ms = ms / args.steps
    per_step_ms = per_traj_ms / wl.steps
    value = job_throughput(world, wl.steps, B, args.steps, ms)
    e2e_value = job_throughput(world, wl.steps, B, args.steps, ms_e2e)
    n_small = int(policy.sum())
    n_large = wl.steps - n_small
    guided = 1 if w == 1.0 else 2
    fl = (n_large * forward_flops(wl.large, guided * B) + n_small * forward_flops(wl.small, guided * B)
          + (text_flops(wl.large, guided * B) if n_large else 0)
          + (text_flops(wl.small, guided * B) if n_small else 0))
    tflops = fl / (per_traj_ms / 1e3) / 1e12

    peaks, src = load_peaks()
    gm, gf, gn = prof["gemm"]
    am, af, an = (a + b for a, b in zip(prof["attention"], prof["cross_attention"]))
    nm = prof["layernorm"][0] + prof["norm_rope"][0]
    nb = prof["layernorm"][1] + prof["norm_rope"][1]
    nn = prof["layernorm"][2] + prof["norm_rope"][2]
    dominant = "gemm" if gm >= am else "attention"
    dm, dflops, dn = prof[dominant]
    achieved = (dflops / dn) / (dm / dn / 1e3) / 1e12 if dn else None
    peak = peaks["bf16_tflops"]
    traffic, traffic_src = measured_traffic("k_gemm_tc" if dominant == "gemm" else "k_attn_pp",
                                            wl.name, dflops / dn if dn else 0.0)
    roof = {"bound": "tensor", "kernel": "bf16 GEMM (tcgen05)" if dominant == "gemm"
            else "flash attention (tcgen05)",
            "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
            "frac": achieved / peak if achieved else None,
            "frac_of_sustained": (achieved / peaks["bf16_tflops_sustained"]
                                  if achieved and peaks.get("bf16_tflops_sustained") else None),
            "traffic": traffic,
            "traffic_unit": "bytes per launch", "traffic_source": traffic_src,
            "peak_source": f"{src} bf16 burst (sustained {peaks.get('bf16_tflops_sustained')})",
            "launches": int(dn), "avg_launch_ms": dm / dn if dn else None,
            "share_of_step": dm / ms_prof if ms_prof else None,
            "measured_in": ("a second pass of the timed steps replaying the trajectory's graph "
                            "recorded with a CUDA event-record node before and after each GEMM, "
                            "attention and norm kernel" if prof_mode == "graph" else
                            "a second pass of the timed steps launched kernel by kernel "
                            "(no graph) with per-launch CUDA events")
                           + f" ({ms_prof / args.steps:.3f} ms/trajectory)",
            "other": {("attention" if dominant == "gemm" else "gemm"):
                      {"ms": am if dominant == "gemm" else gm,
                       "tflops": ((af / (am / 1e3)) if dominant == "gemm" and am
                                  else (gf / (gm / 1e3)) if gm else 0) / 1e12},
                      "norm_kernels": {"ms": nm, "launches": int(nn),
                                       "gb_per_s": (nb / (nm / 1e3) / 1e9) if nm else None,
                                       "frac_of_hbm": ((nb / (nm / 1e3) / 1e9) / peaks["hbm_gbs"])
                                       if nm else None}}}

    cpu = None
    if rank == 0 and not args.skip_cpu:
        sampler = OracleSample(wl)
        sec = sampler.step_seconds(wl.steps - wl.k, wl.k)
        threads, ncpu = cpu_cores()
        cpu = {"value": B / sec, "unit": "steps/s", "cores": threads, "host_cpus": ncpu,
               "kind": "oracle", "sample": sampler.description}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_step_ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": wl.description, "global_batch": world * B,
                       "seq_len": wl.large.tokens, "parallelism": f"replicas x{world}",
                       "l2": "inputs larger than L2: every trajectory streams the large model's "
                             "bf16 weights (2.8 GB for the mid pair) through the 126 MB L2",
                       "policy": "".join("S" if p else "L" for p in policy),
                       "launch": "CUDA graph replay of each trajectory (recorded once per policy)",
                       "timed_unit": f"{args.steps} whole {wl.steps}-step trajectories"},
            "routed_trajectory_ms": per_traj_ms, "all_large_trajectory_ms": ms_all_large / args.steps,
            "speedup_vs_all_large": (ms_all_large / ms) if ms else None,
            "ideal_flop_speedup": wl.steps / (n_large + n_small *
                                              forward_flops(wl.small, 1) / forward_flops(wl.large, 1)),
            "dit_tflops": tflops, "dit_frac_of_bf16_peak": tflops / peak,
            "calibration_ms": calib_ms, "calibration_seeds": wl.calib_seeds,
            "energy": joules,
            "latency_vs_k": sweep,
            "cost_model": {"C_large_ms": c_l, "C_small_ms": c_s, "max_rel_err": cost_err},
            "equal_budget_K": wl.k, "equal_budget": equal_budget,
            "multistep": multistep,
            "score_map": [float(v) for v in q],
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "steps/s",
                    "h2d_bytes_per_step": int(xh.numel() * 4 + ch.numel() * 4 +
                                              (uh.numel() * 4 if uses_uncond else 0)),
                    "d2h_bytes_per_step": int(xh.numel() * 4)},
            "gpu_launches": int(launches),
            "clocks": clocks,
        }
        print(json.dumps(line))
    if world > 1:
        tdist.destroy_process_group()
    return 0




# ---------------------------------------------------------------- one forward of each model
def run_forward(args):
    """One guided denoiser evaluation of each model of a workload at its full size
    (its batch and CFG), timed with CUDA events after warm-up (`--kernel forward`)."""
    import torch

    torch.cuda.set_device(0)
    T = setup_library(args)
    wl = synth.WORKLOADS[args.workload]
    B, w = wl.batch, wl.cfg
    guided = 2 if w != 1.0 else 1
    sig = T.track_schedule(wl.steps, wl.shift)
    x0, c0, u0 = synth.evaluation_inputs(wl.large, 0, B, w != 1.0)
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    sid = stream.cuda_stream
    x = torch.from_numpy(x0).cuda()
    c = torch.from_numpy(c0).cuda()
    u = torch.from_numpy(u0).cuda() if u0 is not None else None
    v = torch.empty_like(x)
    t = float(np.float32(np.float32(1000.0) * np.float32(sig[wl.steps // 2])))
    peaks, src = load_peaks()
    res, clocks = {}, None
    for which, arch, seed in (("large", wl.large, synth.SEED_LARGE),
                              ("small", wl.small, synth.SEED_SMALL)):
        m = T.track_model_create_seeded(arch, seed, T.BF16)
        for _ in range(args.warmup):
            T.track_denoise(m, x, t, c, u, w, v, stream=sid)
        T.track_sync(sid)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with ClockSampler(0) as clk:
            a.record(stream)
            for _ in range(args.steps):
                T.track_denoise(m, x, t, c, u, w, v, stream=sid)
            b.record(stream)
            T.track_sync(sid)
        if which == "large":
            clocks = clk.summary()
        ms = a.elapsed_time(b) / args.steps
        tf = forward_flops(arch, guided * B) / (ms / 1e3) / 1e12
        res[which] = {"ms": ms, "tflops": tf, "frac_of_burst": tf / peaks["bf16_tflops"],
                      "frac_of_sustained": tf / peaks["bf16_tflops_sustained"],
                      "params": synth.param_count(arch)}
        m.close()
        del m
        torch.cuda.empty_cache()
    line = {
        "forward_bench": args.workload, "workload": wl.description, "dtype": "bf16",
        "data": "synthetic", "sequences_per_forward": guided * B,
        "tokens_per_sequence": wl.large.tokens, "steps": args.steps, "warmup": args.warmup,
        "forward_large": res["large"], "forward_small": res["small"],
        "peak_source": src, "clocks": clocks,
    }
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------- HBM-bound kernels
L2_BYTES = 126 * 2 ** 20


def graph_rate(T, torch, stream, make_call, bytes_call, resident_bytes, replays, peaks):
    """Rate of a microsecond-scale HBM kernel: calls recorded back to back in a CUDA
    graph on `stream`, cycling through enough copies of their buffers (make_call()
    makes one) to exceed L2 three times; the replay time over the calls."""
    copies = max(2, math.ceil(3 * L2_BYTES / resident_bytes))
    fns = [make_call() for _ in range(copies)]
    for f in fns:
        f()
    torch.cuda.synchronize()
    reps = max(1, math.ceil(60 / copies))
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for _ in range(reps):
            for f in fns:
                f()
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(replays):
        g.replay()
    e1.record(stream)
    T.track_sync(stream.cuda_stream)
    ms = e0.elapsed_time(e1) / (replays * reps * copies)
    gbs = bytes_call / (ms / 1e3) / 1e9
    del fns, g
    torch.cuda.empty_cache()
    return {"us_per_call": ms * 1e3, "gb_per_s": gbs, "frac_of_hbm": gbs / peaks["hbm_gbs"],
            "bytes_per_call": bytes_call,
            "timing": f"CUDA graph of {reps * copies} calls over {copies} buffer sets"}


def workload_hbm_kernels(T, torch, stream, B, n, peaks):
    """The guidance + Euler update (16 B/elem) and Eq. 4 (8 B/elem) at a workload's
    size (B samples of n latent elements), graph-timed as graph_rate does."""
    def upd():
        fc, fu, xx = (torch.randn(B * n, device="cuda") for _ in range(3))
        return lambda: T.track_cfg_step(xx, fc, fu, 5.0, 0.5, 0.45, stream=stream.cuda_stream)

    def dis():
        pl, ps = (torch.randn(B, n, device="cuda") for _ in range(2))
        acc = torch.zeros(B, device="cuda")
        return lambda: T.track_disagreement(pl, ps, acc, stream=stream.cuda_stream)

    def dis_upd():
        pl, ps, xx = (torch.randn(B, n, device="cuda") for _ in range(3))
        acc = torch.zeros(B, device="cuda")
        return lambda: T.track_disagreement_update(pl, ps, acc, xx, 0.5, 0.45,
                                                   stream=stream.cuda_stream)

    return {"cfg_euler": graph_rate(T, torch, stream, upd, 16.0 * B * n, 12.0 * B * n, 10, peaks),
            "disagreement": graph_rate(T, torch, stream, dis, 8.0 * B * n, 8.0 * B * n, 10, peaks),
            "disagreement_update": graph_rate(T, torch, stream, dis_upd, 16.0 * B * n,
                                              12.0 * B * n, 10, peaks)}


def run_hbm(args, T, torch):
    """The HBM-bound kernels of the C ABI at the sizes the workloads give them, with
    their algorithmic bytes per call: fused guidance + Euler update 16 B/elem (read
    f_c, f_u, x; write x), multistep update 28 B/elem (read x, v and the two history
    arrays; write x and the history), Eq. 4 8 B/elem (read p_L, p_S), its band split
    8 B/elem.  At workload sizes (one 480p request with CFG: 2.1 M latent elements;
    the 4-request serving batch: 8.4 M) a call lasts microseconds, so the calls are
    recorded back to back in a CUDA graph, cycling through enough copies of the
    buffers to exceed L2 three times, and the graph's replay time is divided by the
    calls; the 1 Gi-element case is launched eagerly."""
    peaks, src = load_peaks()
    n480 = 16 * 21 * 60 * 104
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    sg = T.track_schedule(4, 5.0)

    def make(kind, n, B):
        fc, fu, xx = (torch.randn(n, device="cuda") for _ in range(3))
        if kind == "cfg_euler":
            return lambda: T.track_cfg_step(xx, fc, fu, 5.0, 0.5, 0.45)
        if kind == "multistep":
            st = torch.zeros(2 * n, device="cuda")
            T.track_multistep_step(xx, fc, st, sg, 0)          # history for the timed step 1
            return lambda: T.track_multistep_step(xx, fc, st, sg, 1)
        if kind == "disagreement":
            acc = torch.zeros(B, device="cuda")
            return lambda: T.track_disagreement(fc.view(B, -1), fu.view(B, -1), acc)
        if kind == "disagreement_update":
            acc = torch.zeros(B, device="cuda")
            return lambda: T.track_disagreement_update(fc.view(B, -1), fu.view(B, -1), acc,
                                                       xx.view(B, -1), 0.5, 0.45)
        bo = torch.empty(B, 6, device="cuda")
        bl, bs = fc.view(B, 16, 21, 60, 104), fu.view(B, 16, 21, 60, 104)
        return lambda: T.track_band_disagreement(bl, bs, out=bo)

    per_elem = {"cfg_euler": 16.0, "multistep": 28.0, "disagreement": 8.0,
                "disagreement_update": 16.0, "band_split": 8.0}
    resident = {"cfg_euler": 12.0, "multistep": 28.0, "disagreement": 12.0,
                "disagreement_update": 12.0, "band_split": 12.0}   # bytes allocated per element
    out = []
    for label, B in (("one 480p request (latent 16x21x60x104)", 1),
                     ("serving batch of 4 480p requests", 4)):
        for kind in ("cfg_euler", "multistep", "disagreement", "disagreement_update", "band_split"):
            if kind == "band_split" and B != 1:
                continue
            nk = B * n480                # latent elements of the step (per model prediction)
            Bk = B if kind not in ("cfg_euler", "multistep") else 1
            rec = graph_rate(T, torch, stream, lambda: make(kind, nk, Bk), per_elem[kind] * nk,
                             resident[kind] * nk, args.steps, peaks)
            out.append({"kernel": kind, "shape": f"{label}: {nk} elements"
                        + (f", B={Bk}" if Bk > 1 else ""), **rec, "peak_source": src})
    n = 1 << 30
    for kind in ("cfg_euler", "multistep", "disagreement", "disagreement_update"):
        f = make(kind, n, 8)
        for _ in range(args.warmup):
            f()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            f()
        e1.record(stream)
        T.track_sync(stream.cuda_stream)
        ms = e0.elapsed_time(e1) / args.steps
        gbs = per_elem[kind] * n / (ms / 1e3) / 1e9
        out.append({"kernel": kind, "shape": f"1 Gi elements{', B=8' if 'disagree' in kind else ''}",
                    "us_per_call": ms * 1e3, "gb_per_s": gbs, "frac_of_hbm": gbs / peaks["hbm_gbs"],
                    "timing": "eager launches", "peak_source": src})
        del f
        torch.cuda.empty_cache()
    print(json.dumps({"kernel_bench": "hbm", "results": out}))
    return 0


# ---------------------------------------------------------------- single kernels
GEMM_SCHEDULES = {"auto": 0, "dp": 1, "sk": 2}   # track_gemm/attention_schedule modes


def run_kernel(args):
    """Times one kernel class alone at the workload's shapes (large model, `--batch`
    sequences): the GEMMs of one block, or self- and cross-attention."""
    import torch

    torch.cuda.set_device(0)
    T = setup_library(args)
    wl = synth.WORKLOADS[args.workload]
    a = wl.large
    M = args.batch * a.tokens
    d, F, H, hd = a.dim, a.ffn, a.heads, a.head_dim
    g = torch.Generator(device="cuda").manual_seed(0)
    rnd = lambda *shape: (torch.randn(*shape, device="cuda", generator=g) * 0.5).to(torch.bfloat16)
    cases = []
    if args.kernel == "gemm":
        for name, N, K, epi in (("qkv", 3 * d, d, T.EPI_STORE), ("out_proj", d, d, T.EPI_RESID_GATE),
                                ("cross_q", d, d, T.EPI_STORE),
                                ("ffn_up", F, d, T.EPI_GELU), ("ffn_down", d, F, T.EPI_RESID_GATE)):
            X, W = rnd(M, K), rnd(N, K)
            b = torch.zeros(N, device="cuda")
            gate = torch.ones(N, device="cuda")
            out = (torch.zeros(M, N, device="cuda", dtype=torch.bfloat16) if epi in (0, 1)
                   else torch.zeros(M, N, device="cuda"))
            fn = (lambda X=X, W=W, b=b, epi=epi, out=out, gate=gate:
                  T.track_linear(T.BF16, X, W, b, epi, out, gate=gate if epi == 2 else None))
            cases.append((name, f"M={M} N={N} K={K}", 2.0 * M * N * K, fn))
    elif args.kernel == "attention":
        Q, Kt, V = (rnd(args.batch, H, a.tokens, hd) for _ in range(3))
        Kc, Vc = rnd(args.batch, H, a.text_len, hd), rnd(args.batch, H, a.text_len, hd)
        O = torch.empty(args.batch, a.tokens, H, hd, device="cuda", dtype=torch.bfloat16)
        cases.append(("self_attention", f"S={args.batch} H={H} L={a.tokens} hd={hd}",
                      4.0 * args.batch * H * a.tokens * a.tokens * hd,
                      lambda: T.track_attention(T.BF16, Q, Kt, V, O)))
        cases.append(("cross_attention", f"S={args.batch} H={H} Lq={a.tokens} Lk={a.text_len}",
                      4.0 * args.batch * H * a.tokens * a.text_len * hd,
                      lambda: T.track_attention(T.BF16, Q, Kc, Vc, O)))
    elif args.kernel == "hbm":
        return run_hbm(args, T, torch)
    peaks, src = load_peaks()
    out = []
    for name, shape, flops, fn in cases:
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.steps):
            fn()
        e1.record()
        T.track_sync()
        ms = e0.elapsed_time(e1) / args.steps
        tf = flops / (ms / 1e3) / 1e12
        out.append({"kernel": name, "shape": shape, "ms": ms, "tflops": tf,
                    "frac_of_burst": tf / peaks["bf16_tflops"],
                    "frac_of_sustained": tf / peaks["bf16_tflops_sustained"], "peak_source": src})
    print(json.dumps({"kernel_bench": args.kernel, "workload": wl.description, "batch": args.batch,
                      "results": out}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(synth.WORKLOADS), default=WORKLOAD,
                    help="the configuration (default: the Wan-2.1-shaped 480p pair)")
    ap.add_argument("--skip-cpu", action="store_true", help="omit the oracle CPU baseline")
    ap.add_argument("--no-trajectories", action="store_true",
                    help="omit the whole routed and all-large trajectories")
    ap.add_argument("--profile-steps", type=int, default=6,
                    help="timed steps run again with per-kernel events")
    ap.add_argument("--calibrate", action="store_true",
                    help="run the workload's calibration and write its score map")
    ap.add_argument("--seeds", type=int, default=0, help="calibration samples (default: the workload's)")
    ap.add_argument("--calib-batch", type=int, default=0, help="calibration samples per call")
    ap.add_argument("--fresh", action="store_true", help="recalibrate from the first sample")
    ap.add_argument("--kernel", choices=["gemm", "attention", "hbm", "forward"], default=None,
                    help="time one kernel class (or one forward of each model) alone")
    ap.add_argument("--batch", type=int, default=1, help="sequences for --kernel")
    ap.add_argument("--gemm-schedule", choices=["auto", "dp", "sk"], default="auto",
                    help="bf16 GEMM schedule: makespan model, data-parallel or stream-K")
    ap.add_argument("--attn-schedule", choices=["auto", "dp", "sk"], default="auto",
                    help="bf16 attention schedule: makespan model, data-parallel or stream-K")
    ap.add_argument("--gemm-raster", type=int, default=0,
                    help="bf16 GEMM raster group in 128-row units (0: the default)")
    ap.add_argument("--attn-one-tile", action="store_true",
                    help="attention work items of one query tile instead of a pair")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)     # at least three untimed warm-up steps
    if args.impl == "reference":
        return run_reference(args)
    if args.calibrate:
        return run_calibrate(args)
    if args.kernel == "forward":
        return run_forward(args)
    if args.kernel:
        return run_kernel(args)
    if args.workload in WINDOW_WORKLOADS:
        return run_window(args)
    return run_trajectories(args)


if __name__ == "__main__":
    sys.exit(main())
