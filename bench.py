"""NGFF throughput on GB300: frames/s and pixel GB/s of the whole filtering
path (histogram kernel + windowed-distance kernel + scan kernel) over the
1080p stream (3600 uint8 RGB frames of 1920x1080, one whole-stream push).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

One step = reset the stream, then push all 3600 frames through the library
and decide every frame. Inputs (22.4 GB per step) are larger than L2, so no
flush is needed between steps. Prints one JSON line (rank 0).

Under torchrun each rank filters its own independently seeded 1080p stream
(weak scaling, no collective on the data path); timing is the max over
ranks. ``--impl reference`` times the single-threaded C oracle on the host
cores on a bounded sample of the same stream (rank 0 only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

REPO = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, REPO)

METRIC = "NGFF frames/s and pixel GB/s (fraction of HBM peak) at 1 GB300 vs CPU oracle"
UNIT = "frames/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
K1_SOURCES = [os.path.join(REPO, "paper_2609_03675_gb300", "csrc", f)
              for f in ("ngff_hist.cu", "ngff_device.cuh", "ngff_common.cuh")]
K1_TRAFFIC = os.path.join(REPO, "profiles", "k1_hist_1080p_traffic.json")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=600)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--e2e-steps", type=int, default=7)
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="target CPU work of the oracle baseline")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--workload", choices=["hd1080", "serving", "medium", "rare_event", "gather", "qer", "shards",
                                           "signals", "pipeline", "tiny", "static", "sensitivity"],
                    default="hd1080",
                    help="hd1080 is the benchmark line; the others print their own JSON lines (latency, recall, "
                         "finalize + gather bandwidth)")
    ap.add_argument("--qer-frames", type=int, default=128, help="candidate frames of the qer workload")
    ap.add_argument("--qer-kernel", type=int, default=0, choices=[0, 1, 2],
                    help="qer scoring kernel: 0 automatic, 1 one-SM, 2 paired-SM")
    ap.add_argument("--l-max", type=int, default=30,
                    help="L_max of the hd1080 workload (0: no forced retention, the rule walked in frame order)")
    ap.add_argument("--signal", choices=["histogram", "lowres", "dhash", "scd"], default="histogram",
                    help="NGFF's novelty signal for the hd1080 workload (histogram is the paper's)")
    ap.add_argument("--frames", type=int, default=3600,
                    help="use the first FRAMES frames of the stream (small cases for profiling; default all 3600)")
    ap.add_argument("--no-configs", action="store_true",
                    help="hd1080 line without the figures of the tiny, medium, serving and rare-event streams")
    ap.add_argument("--configs-budget", type=float, default=240.0,
                    help="seconds the other streams' figures may take after the headline (a config that would start "
                         "past the budget is skipped and says so)")
    ap.add_argument("--no-parity", action="store_true", help="hd1080 line without the oracle parity block")
    ap.add_argument("--serving-frames", type=int, default=0,
                    help="frames per stream of the serving workload (0: all 1800; fewer for profiling captures)")
    ap.add_argument("--size", default="1920x1080",
                    help="frame size WxH of the hd1080 workload's stream (same recipe); a pixel count that is not a "
                         "multiple of 16 runs the generic histogram kernel")
    return ap.parse_args()


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def stream_seed(rank: int) -> int:
    """Each rank filters its own independently seeded 1080p stream."""
    import synth
    return synth.SEED_BASE + 3 + rank


def max_over_ranks(x: float, device="cuda") -> float:
    """The largest value of x over all ranks (a no-op without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, world: int, seconds_max: float) -> float:
    """Whole-job throughput: the units all ranks processed over the slowest rank's time."""
    return units_per_rank * world / seconds_max


def peaks():
    try:
        with open(os.path.join(REPO, "MEASURED_PEAKS.json")) as fh:
            d = json.load(fh)
        return float(d["hbm_gbs"]), "measured"
    except Exception:  # noqa: BLE001 -- file absent: the recipe's fallback
        return FALLBACK_HBM_GBS, "fallback"


def k1_source_hash() -> str:
    """sha256 over K1's sources (the kernel file, its device helpers, and the common header)."""
    h = hashlib.sha256()
    for path in K1_SOURCES:
        h.update(open(path, "rb").read())
    return h.hexdigest()


def k1_traffic_per_launch():
    """DRAM bytes per histogram launch from the committed ncu summary, or None
    when the kernel source changed since the counters were taken."""
    try:
        with open(K1_TRAFFIC) as fh:
            d = json.load(fh)
        src = k1_source_hash()
        if d.get("source_sha256") != src:
            return None
        return float(d["dram_bytes_per_launch_full"])
    except Exception:  # noqa: BLE001
        return None


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.proc = None
        self.gpu_id = gpu_id

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        self.file.flush()
        self.file.seek(0)
        rows = [ln.strip().split(", ") for ln in self.file.read().splitlines() if ln.strip()]
        os.unlink(self.file.name)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[0]))
                mx = float(r[1])
                for name, v in zip(names, r[4:8]):
                    if v.strip().lower() == "active":
                        reasons.add(name)
            except (ValueError, IndexError):
                continue
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


SIGNALS = {"histogram": 0, "lowres": 1, "dhash": 2, "scd": 3}


def oracle_sample(frames_u8_ptr, spec, target_s: float, signal: int = 0, l_max: int = 30):
    """The oracle as it stands (single-threaded C for the histogram, numpy for
    the spatial signals) on the first k frames of the stream; k sized to about
    target_s seconds of CPU work."""
    import ctypes

    import numpy as np

    import oracle as O
    from oracle import scd_oracle as SC
    from oracle import signals_oracle as SO
    o = O.load()
    p = O.Params(spec.width, spec.height, l_max=l_max)
    fb = spec.frame_bytes

    def run(k):
        arr = np.ctypeslib.as_array((ctypes.c_uint8 * (k * fb)).from_address(frames_u8_ptr))
        t = time.perf_counter()
        if signal == 3:
            SC.run(arr.reshape(k, spec.height, spec.width, 3), p, 0.30, 0.10)
        elif signal:
            SO.run(arr.reshape(k, spec.height, spec.width, 3), p, signal)
        else:
            o.run(arr.reshape(k, spec.height, spec.width, 3), p)
        return time.perf_counter() - t

    t2 = run(2)
    k = int(max(2, min(spec.frames, target_s / max(t2 / 2, 1e-6))))
    dt = run(k)
    return k, dt


def oracle_parallel_sample(frames_u8_ptr, spec, target_s: float, l_max: int = 30):
    """The oracle's histogram routine mapped over all host cores (frames in
    parallel), then its selection, on the first k frames; k sized to about
    target_s seconds. Returns (k, seconds, cores)."""
    import oracle as O
    o = O.load()
    p = O.Params(spec.width, spec.height, l_max=l_max)
    cores = max(1, len(os.sched_getaffinity(0)))

    def run(k):
        t = time.perf_counter()
        hist = o.histograms_parallel(frames_u8_ptr, k, p, nthreads=cores)
        o.select(hist, p)
        return time.perf_counter() - t

    t1 = run(min(cores, spec.frames))
    per = t1 / min(cores, spec.frames)
    k = int(max(cores, min(spec.frames, target_s / max(per, 1e-6))))
    return k, run(k), cores


SCORE_RTOL = 1e-6  # the fp32 score against the oracle's double-precision distance
SERVING_E2E_FRAMES = 300  # frames per stream of the serving workload's end-to-end leg (6.6 GB of pinned frames)


def parity_block(tau, scores, keep, want_scores, want_keep, hist=None, want_hist=None, idx=None, want_idx=None):
    """Oracle parity of one run: histograms bit-exact, keep codes identical,
    the largest relative score error, and the frames whose oracle score lies
    within the score tolerance of tau_h (the band where the keep decision
    could legitimately differ; listed even when every decision agrees)."""
    import numpy as np
    sg = np.asarray(scores, dtype=np.float64)
    so = np.asarray(want_scores, dtype=np.float64)
    rel = np.abs(sg - so) / np.maximum(np.abs(so), 1e-300)
    rel[(so == 0) & (sg == 0)] = 0.0
    band = np.flatnonzero(np.abs(so - tau) <= SCORE_RTOL * max(abs(tau), 1e-30))
    diff = np.flatnonzero(np.asarray(keep) != np.asarray(want_keep))
    out = {"frames": int(so.size), "keep_equal": bool(diff.size == 0),
           "keep_mismatch_outside_band": int(np.setdiff1d(diff, band).size),
           "max_rel_score_err": float(rel.max()) if rel.size else 0.0, "score_rtol": SCORE_RTOL,
           "band_frames": [int(x) for x in band[:64]], "band_count": int(band.size)}
    if want_hist is not None:
        out["hist_equal"] = bool(hist is not None and np.array_equal(np.asarray(hist), np.asarray(want_hist)))
    if want_idx is not None:
        out["candidates_equal"] = bool(idx is not None and np.array_equal(np.asarray(idx, dtype=np.uint32),
                                                                           np.asarray(want_idx, dtype=np.uint32)))
    return out


def _event_runs(ev):
    runs, t = [], 0
    while t < ev.size:
        if ev[t]:
            u = t
            while u < ev.size and ev[u]:
                u += 1
            runs.append((t, u))
            t = u
        else:
            t += 1
    return runs


def tiny_figures(args):
    """The tiny stream (64 uint8 RGB frames of 224x224, one whole-stream push):
    device-resident frames/s from CUDA events over repeated steps, per-push
    latency (host call + synchronise), end to end from pinned host frames to
    host outputs through the same C entry point, and oracle parity."""
    import numpy as np
    import torch

    import oracle as O
    import synth
    from paper_2609_03675_gb300 import NGFF
    spec = synth.tiny()
    T = spec.frames
    host = torch.empty((T, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.cuda()
    f = NGFF(spec.width, spec.height)
    scores = torch.empty(T, dtype=torch.float32, device="cuda")
    keep = torch.empty(T, dtype=torch.uint8, device="cuda")

    def step():
        f.reset()
        f.push(dev, scores=scores, keep=keep)

    for _ in range(20):
        step()
    torch.cuda.synchronize()
    reps = 300
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        step()
    e1.record()
    torch.cuda.synchronize()
    dev_s = e0.elapsed_time(e1) / 1e3
    lat = []
    for _ in range(200):
        c0 = time.perf_counter()
        step()
        torch.cuda.synchronize()
        lat.append((time.perf_counter() - c0) * 1e3)
    hs = torch.empty(T, dtype=torch.float32, pin_memory=True)
    hk = torch.empty(T, dtype=torch.uint8, pin_memory=True)
    e2e = []
    for i in range(60):
        torch.cuda.synchronize()
        c0 = time.perf_counter()
        f.reset()
        f.push(host, scores=hs, keep=hk)
        torch.cuda.synchronize()
        if i >= 10:
            e2e.append(time.perf_counter() - c0)
    f.reset()
    s, k, h = f.push(dev, return_hist=True)
    idx = f.candidates(0)
    f.status()
    o = O.load()
    ho, so, ko = o.run(host.numpy(), O.Params(spec.width, spec.height))
    par = parity_block(0.30, s.cpu().numpy(), k.cpu().numpy(), so, ko, h.cpu().numpy().view(np.uint32), ho,
                       idx.cpu().numpy(), o.candidates(ko, 4))
    assert torch.equal(hk, k.cpu()), "end-to-end keep codes differ from the device-resident run"
    f.close()
    e2e_s = statistics.median(e2e)
    return {"workload": "tiny: 64 uint8 RGB frames of 224x224, one whole-stream push per step, B=32, L_max=30, "
                        "tau_h=0.30",
            "frames_per_s": reps * T / dev_s, "ms_per_step": dev_s / reps * 1e3,
            "pixel_gbs": reps * T * spec.frame_bytes / dev_s / 1e9,
            "latency_ms_p50": _pct(lat, 50), "latency_ms_p99": _pct(lat, 99),
            "e2e": {"frames_per_s": T / e2e_s, "ms_per_step": e2e_s * 1e3, "h2d_bytes_per_step": T * spec.frame_bytes,
                    "d2h_bytes_per_step": T * 5, "statistic": "median of 50 steps"},
            "kept": int((k != 0).sum().item()), "parity": par,
            "timing": f"CUDA events over {reps} steps (reset + push); latency: host call + synchronise, 200 steps"}


def hd1080_parity(f, dev, host, spec, signal, l_max):
    """Parity of the benchmark's own configuration (same handle, same frames
    as the timed steps): GPU histograms, scores, keep codes and the stream's
    candidate set against the oracle. For the spatial signals, whose oracle
    is numpy per frame, this is left to the tests."""
    import numpy as np

    import oracle as O
    from oracle import scd_oracle as SC
    if signal in (1, 2):
        return {"skipped": "the spatial signals' oracle is numpy per frame; their parity is in the GPU tests"}
    t0 = time.perf_counter()
    T = spec.frames
    f.reset()
    s, k, h = f.push(dev, return_hist=True)
    idx = f.candidates(0)
    f.status()
    o = O.load()
    p = O.Params(spec.width, spec.height, l_max=l_max)
    cores = max(1, len(os.sched_getaffinity(0)))
    hist_o = o.histograms_parallel(host.data_ptr(), T, p, nthreads=cores)
    so, ko = SC.select(hist_o, p, 0.30, 0.10) if signal == 3 else o.select(hist_o, p)
    out = parity_block(0.30, s.cpu().numpy(), k.cpu().numpy(), so, ko, h.cpu().numpy().view(np.uint32), hist_o,
                       idx.cpu().numpy(), o.candidates(ko, 4))
    out["oracle"] = (f"C oracle histograms on {cores} host threads (frames in parallel), then its selection "
                     "rule and candidate set, single-threaded")
    out["seconds"] = time.perf_counter() - t0
    return out


def _compact(x, digits=5):
    """x with floats rounded to `digits` significant digits (a short line)."""
    if isinstance(x, float):
        return float(f"{x:.{digits}g}")
    if isinstance(x, dict):
        return {k: _compact(v, digits) for k, v in x.items()}
    if isinstance(x, list):
        return [_compact(v, digits) for v in x]
    return x


def _config_summary(name, d):
    """The figures of one config kept in the headline line (the full figures
    are printed by bench.py --workload NAME)."""
    keep = {"tiny": ("workload", "frames_per_s", "ms_per_step", "pixel_gbs", "latency_ms_p50", "latency_ms_p99", "e2e",
                     "kept", "parity"),
            "medium": ("workload", "pipelined_frames_per_s", "graph_frames_per_s", "graph_ms_per_push",
                       "latency_ms_p50", "latency_ms_p99", "e2e", "kernels_per_push", "kept", "parity"),
            "serving": ("workload", "calls", "pipelined_frames_per_s", "graph_frames_per_s", "graph_ms_per_call",
                        "latency_ms_p50", "latency_ms_p99", "keep_ratio", "e2e", "parity"),
            "rare_event": ("workload", "frames_per_s", "pixel_gbs", "events", "e2e", "taus")}[name]
    out = {k: d[k] for k in keep if k in d}
    if name == "rare_event":  # per tau: keep ratio, event-frame recall, per-event recall; one parity summary
        taus = out.pop("taus")
        out["recall_by_tau"] = {t: [v["keep_ratio"], v["event_frame_recall"], v["event_recall"]] for t, v in taus.items()}
        out["recall_fields"] = ["keep_ratio", "event_frame_recall", "event_recall"]
        out["parity"] = {"keep_equal_every_tau": all(v["parity"]["keep_equal"] for v in taus.values()),
                         "max_rel_score_err": max(v["parity"]["max_rel_score_err"] for v in taus.values()),
                         "band_frames": sorted({f for v in taus.values() for f in v["parity"]["band_frames"]})}
    for e in ("e2e",):
        if isinstance(out.get(e), dict):
            out[e] = {k: v for k, v in out[e].items() if k not in ("how", "statistic")}
    par = out.get("parity")
    if isinstance(par, dict):
        out["parity"] = {k: v for k, v in par.items() if k in ("frames", "hist_equal", "keep_equal", "keep_equal_every_tau",
                                                                 "keep_mismatch_outside_band", "max_rel_score_err",
                                                                 "band_frames", "candidates_equal")}
    if "seconds" in d:
        out["seconds"] = d["seconds"]
    return _compact(out)


def other_configs(args):
    """Figures of the benchmark's other streams, each at its full size, in one
    run after the headline: tiny (64 x 224x224), medium (600 x 448x448 in
    pushes of 8), rare-event (3600 x 1280x720) and serving (32 x 1800 x
    640x360). A config that would start after args.configs_budget seconds is
    skipped and says so."""
    import torch
    t_start = time.perf_counter()
    out = {}
    for name, fn in (("tiny", tiny_figures), ("medium", medium_figures), ("rare_event", rare_event_figures),
                     ("serving", serving_figures)):
        el = time.perf_counter() - t_start
        if el > args.configs_budget:
            out[name] = {"skipped": f"the {args.configs_budget:.0f} s budget was spent ({el:.0f} s)"}
            continue
        t0 = time.perf_counter()
        d = fn(args)
        d["seconds"] = time.perf_counter() - t0
        out[name] = _config_summary(name, d)
        torch.cuda.empty_cache()
    out["seconds"] = round(time.perf_counter() - t_start, 1)
    return out


def bench_gb300(args):
    import numpy as np  # noqa: F401
    import torch
    import torch.distributed as dist

    import synth
    from paper_2609_03675_gb300 import NGFF

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    spec = synth.hd1080(seed=stream_seed(rank))
    sw, sh = (int(x) for x in args.size.lower().split("x"))
    spec = spec.with_(frames=min(spec.frames, max(1, args.frames)), width=sw, height=sh)
    T = spec.frames
    # inputs: generated on the host (pinned, kept for the end-to-end leg), resident in HBM for the timed region
    host = torch.empty((T, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.to("cuda", non_blocking=True)
    scores = torch.empty(T, dtype=torch.float32, device="cuda")
    keep = torch.empty(T, dtype=torch.uint8, device="cuda")
    signal = SIGNALS[args.signal]
    f = NGFF(spec.width, spec.height, max_frames_per_push=T, signal=signal, l_max=args.l_max)
    stream = torch.cuda.current_stream()

    def step():
        f.reset()
        f.push(dev, scores=scores, keep=keep)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    f.status()

    props = torch.cuda.get_device_properties(local)
    gpu_id = "GPU-" + str(props.uuid) if getattr(props, "uuid", None) else str(local)
    f.profile_reset(time_kernels=True)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu_id) as clk:
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        start.record(stream)
        for _ in range(args.steps):
            step()
        end.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
    f.status()
    prof = f.profile_read()
    ms = max_over_ranks(start.elapsed_time(end))
    clocks = clk.summary()
    clocks["gpu_uuid"] = gpu_id
    kept = int((keep != 0).sum().item())

    frames_total = args.steps * T * world
    value = whole_job_rate(args.steps * T, world, ms / 1e3)
    pixel_gbs = frames_total * spec.frame_bytes / (ms / 1e3) / 1e9

    # roofline of the dominant kernel (histogram): algorithmic bytes per launch / mean event-timed duration
    peak, peak_kind = peaks()
    k1_ms = prof["hist_ms"] / max(prof["hist_timed"], 1)
    k1_bytes = prof["hist_bytes"] / max(prof["hist_launches"], 1)
    achieved = k1_bytes / (k1_ms / 1e3) / 1e9
    traffic = k1_traffic_per_launch() if signal == 0 and (spec.width, spec.height) == (1920, 1080) else None

    # end to end through the same C entry point with host buffers: H2D of the
    # step's frames and D2H of its scores and keep codes inside the timed region
    e2e = None
    if not args.no_e2e:
        hs = torch.empty(T, dtype=torch.float32, pin_memory=True)
        hk = torch.empty(T, dtype=torch.uint8, pin_memory=True)
        fe = NGFF(spec.width, spec.height, max_frames_per_push=T, signal=signal, l_max=args.l_max)

        def estep():
            fe.reset()
            fe.push(host, scores=hs, keep=hk)

        for _ in range(2):  # untimed: the first passes over the pinned buffer are the slowest
            estep()
        torch.cuda.synchronize()
        # the raw host->device link over the same bytes (one plain copy of the
        # whole pinned stream into the device frame tensor), measured right
        # before and right after the end-to-end steps, to read the e2e figure against
        def link():
            torch.cuda.synchronize()
            tl = time.perf_counter()
            dev.copy_(host, non_blocking=True)
            torch.cuda.synchronize()
            return host.numel() / (time.perf_counter() - tl) / 1e9

        link_before = link()
        if world > 1:
            dist.barrier()
        step_s = []
        for _ in range(args.e2e_steps):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            estep()
            torch.cuda.synchronize()
            step_s.append(time.perf_counter() - t0)
        # the host link of this machine shows sporadic multi-fold slowdowns (plain
        # copies included), so the reported step is the median over steps
        el = max_over_ranks(statistics.median(step_s))
        link_after = link()
        fe.status()
        assert torch.equal(hk.to("cuda"), keep), "end-to-end keep codes differ from the device-resident run"
        e2e = {"value": whole_job_rate(T, world, el), "unit": UNIT,
               "h2d_bytes_per_step": T * spec.frame_bytes, "d2h_bytes_per_step": T * (4 + 1),
               "ms_per_step": el * 1e3, "ms_per_step_min": min(step_s) * 1e3, "ms_per_step_max": max(step_s) * 1e3,
               "statistic": f"median of {args.e2e_steps} steps", "h2d_link_gbs_before": link_before,
               "h2d_link_gbs_after": link_after,
               "h2d_achieved_gbs": T * spec.frame_bytes / el / 1e9}
        fe.close()

    # oracle parity of the timed configuration: one more step with the
    # histograms out, against the oracle's histograms (its routine on all host
    # cores) and its selection on them
    parity = None
    if rank == 0 and not args.no_parity:
        parity = hd1080_parity(f, dev, host, spec, signal, args.l_max)
    cpu = None
    if rank == 0 and world == 1 and args.cpu_seconds > 0:
        k, dt = oracle_sample(host.data_ptr(), spec, args.cpu_seconds, signal, args.l_max)
        what = {0: "single-threaded C oracle (histograms + selection)",
                3: "C oracle histograms + the scene-change oracle's rule (Python)"}.get(
            signal, f"numpy signals oracle ({args.signal} features + selection)")
        cpu = {"value": k / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"first {k} frames of the 1080p stream, {what}",
               "wall_s": dt, "pixel_gbs": k * spec.frame_bytes / dt / 1e9}
        if signal == 0:
            kp, dtp, cores = oracle_parallel_sample(host.data_ptr(), spec, args.cpu_seconds / 2, args.l_max)
            cpu["all_cores"] = {"value": kp / dtp, "unit": UNIT, "cores": cores, "wall_s": dtp,
                                "pixel_gbs": kp * spec.frame_bytes / dtp / 1e9,
                                "sample": f"first {kp} frames, the oracle's histogram routine on {cores} threads "
                                          "(frames in parallel), then its selection"}

    # the other streams of the benchmark, after everything above (rank 0 at N=1)
    configs = None
    if rank == 0 and world == 1 and not args.no_configs:
        f.close()
        del dev, host
        torch.cuda.empty_cache()
        configs = other_configs(args)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "u8", "data": "synthetic",
            "config": {"workload": f"1080p stream: {T} uint8 RGB frames of {spec.width}x{spec.height} (HWC), one "
                                   f"whole-stream push per step, B=32, L_max={args.l_max}, tau_h=0.30"
                                   + ("" if signal == 0 else f", signal {args.signal} in place of the histogram"),
                       "signal": args.signal, "frames_per_step": T, "width": spec.width, "height": spec.height,
                       "bins": 32, "l_max": args.l_max,
                       "tau": 0.30, "l2": f"inputs larger than L2 ({T * spec.frame_bytes / 1e9:.1f} GB per step), no flush",
                       "parallelism": f"{world} independent stream(s), one per GPU"},
            "pixel_gbs": pixel_gbs,
            "frac_of_nominal_8tbs": pixel_gbs / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "peak_kind": f"{peak_kind} copy bandwidth", "traffic": traffic,
                         "kernel": ("ngff histogram (K1)" if (spec.width * spec.height) % 16 == 0
                                    else "ngff histogram, generic kernel (pixel count not a multiple of 16)")
                         if signal == 0 else f"ngff {args.signal} cell sums (K1 cells)",
                         "launch_ms": k1_ms, "bytes_per_launch": k1_bytes,
                         "select_ms_per_step": prof["select_ms"] / max(prof["select_timed"], 1)},
            "e2e": e2e,
            "cpu_baseline": cpu,
            "gpu_launches": int(prof["hist_launches"] + prof["select_launches"] + prof["other_launches"]),
            "clocks": clocks,
            "kept_frames_last_step": kept,
            "parity": parity,
            "configs": configs,
        }
        for k in ("pixel_gbs", "frac_of_nominal_8tbs", "roofline", "e2e", "cpu_baseline", "parity"):
            line[k] = _compact(line[k], 6)
        print(json.dumps(line), flush=True)
    f.close()
    if world > 1:
        dist.destroy_process_group()


def bench_reference(args):
    """The oracle (single-threaded C, host cores) on the same workload and
    metric: the timed steps cover the 3600-frame 1080p stream in consecutive
    slices of about T / K frames (at most 200 per step, so K >= 18 covers the
    whole stream), each
    slice a stream the oracle filters from its first frame; the warm-up steps
    run an 8-frame sample."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import oracle as O
    import synth
    spec = synth.hd1080()
    o = O.load()
    p = O.Params(spec.width, spec.height)
    T = spec.frames
    steps = max(1, args.steps)
    per_step = min(200, -(-T // steps))
    import numpy as np
    buf = np.empty((per_step, spec.height, spec.width, 3), dtype=np.uint8)
    warm = synth.generate(spec, 0, 8)
    for _ in range(args.warmup):
        o.run(warm, p)
    el, done = 0.0, 0
    for i in range(steps):
        a = (i * per_step) % T
        b = min(a + per_step, T)
        synth.generate(spec, a, b, out=buf)
        t0 = time.perf_counter()
        o.run(buf[: b - a], p)
        el += time.perf_counter() - t0
        done += b - a
    value = done / el
    sample = (f"{steps} consecutive slices of up to {per_step} frames of the 1080p stream ({done} frames"
              f"{', the whole stream' if done >= T else ''}), single-threaded C oracle (histograms + selection)")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": el / steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u8", "data": "synthetic",
        "config": {"workload": "1080p stream: 3600 uint8 RGB frames of 1920x1080 (HWC), B=32, L_max=30, tau_h=0.30",
                   "frames_per_step": per_step, "frames_timed": done, "width": spec.width, "height": spec.height},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample,
                         "wall_s": el},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def _pct(xs, q):
    import numpy as np
    return float(np.percentile(np.asarray(xs), q))


def _graph_seconds(capture, reset, reps=5):
    """Wall seconds of one launch of a CUDA graph holding a whole sequence of
    pushes (captured once by `capture`), best of `reps` after one untimed
    launch; `reset` restarts the streams before each launch, outside the graph."""
    import torch
    g = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        capture()
    times = []
    for _ in range(reps + 1):
        reset()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        g.replay()
        torch.cuda.synchronize()
        times.append(time.perf_counter() - t0)
    return min(times[1:])


def bench_serving(args):
    print(json.dumps(serving_figures(args)), flush=True)


def serving_figures(args, parity: bool = True):
    """32 concurrent 640x360 streams, each call pushing U{1..8} new frames per
    stream in one batched launch sequence: per-call latency (synchronised
    calls) and pipelined aggregate frames/s; the pipelined run's keep codes
    and scores against the oracle (its histogram routine on all host cores)."""
    import numpy as np
    import torch

    import oracle as O
    import synth
    from paper_2609_03675_gb300 import NGFF
    S = synth.SERVING_STREAMS
    specs = [synth.serving_stream(s) for s in range(S)]
    if getattr(args, "serving_frames", 0):
        specs = [sp.with_(frames=min(sp.frames, args.serving_frames)) for sp in specs]
    T, W, H = specs[0].frames, specs[0].width, specs[0].height
    host = torch.empty((T, H, W, 3), dtype=torch.uint8, pin_memory=True)
    dev, want = [], []
    o = O.load()
    p = O.Params(W, H)
    for sp in specs:
        synth.generate(sp, out=host.data_ptr())
        dev.append(host.cuda())
        if parity:
            want.append(o.select(o.histograms_parallel(host.data_ptr(), T, p), p))
    del host
    sizes = [synth.push_sizes(synth.SEED_BASE + 4, s, T) for s in range(S)]
    scores = torch.empty((S, T), dtype=torch.float32, device="cuda")
    keep = torch.empty((S, T), dtype=torch.uint8, device="cuda")
    f = NGFF(W, H, max_streams=S)

    def calls():
        pos, call, out = [0] * S, 0, []
        while min(pos) < T:
            items = []
            for s in range(S):
                if pos[s] >= T:
                    continue
                n = int(min(sizes[s][call], T - pos[s]))
                items.append((s, dev[s][pos[s]:pos[s] + n], scores[s, pos[s]:pos[s] + n], keep[s, pos[s]:pos[s] + n]))
                pos[s] += n
            out.append(items)
            call += 1
        return out

    plan = [f.make_batch(items) for items in calls()]  # descriptors marshalled once, outside the timing
    frames_total = S * T
    st = torch.cuda.current_stream().cuda_stream

    def run(sync_each):
        for s in range(S):
            f.reset(s)
        lat = []
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for arr, nd in plan:
            c0 = time.perf_counter()
            f.push_batch_raw(arr, nd, st)
            if sync_each:
                torch.cuda.synchronize()
                lat.append((time.perf_counter() - c0) * 1e3)
        torch.cuda.synchronize()
        return time.perf_counter() - t0, lat

    for _ in range(max(1, args.warmup // 3)):
        run(False)
    el_pipe, _ = run(False)
    f.status()
    par = None
    if parity:
        sc, kc = scores.cpu().numpy(), keep.cpu().numpy()
        par = parity_block(0.30, sc.reshape(-1), kc.reshape(-1), np.concatenate([w[0] for w in want]),
                           np.concatenate([w[1] for w in want]))
        par["candidates_equal"] = all(
            np.array_equal(f.candidates(s).cpu().numpy().astype(np.uint32), o.candidates(want[s][1], 4))
            for s in range(S))
        par["streams"] = S
    el_sync, lat = run(True)
    f.status()

    def reset_all():
        for s in range(S):
            f.reset(s)

    el_graph = _graph_seconds(lambda: [f.push_batch_raw(arr, nd) for arr, nd in plan], reset_all)
    f.status()

    # end to end: the same calls over the first E frames of every stream with
    # the frames in pinned host memory and the scores and keep codes written
    # to pinned host memory, through the same batched entry point
    E = min(T, SERVING_E2E_FRAMES)
    host_fr = torch.empty((S, E, H, W, 3), dtype=torch.uint8, pin_memory=True)
    for s in range(S):
        host_fr[s].copy_(dev[s][:E])
    hs = torch.empty((S, E), dtype=torch.float32, pin_memory=True)
    hk = torch.empty((S, E), dtype=torch.uint8, pin_memory=True)
    hplan, pos, call = [], [0] * S, 0
    while min(pos) < E:
        items = []
        for s in range(S):
            if pos[s] >= E:
                continue
            n = int(min(sizes[s][call], E - pos[s]))
            items.append((s, host_fr[s, pos[s]:pos[s] + n], hs[s, pos[s]:pos[s] + n], hk[s, pos[s]:pos[s] + n]))
            pos[s] += n
        hplan.append(f.make_batch(items))
        call += 1
    torch.cuda.synchronize()

    def run_host(sync_each):
        reset_all()
        hlat = []
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for arr, nd in hplan:
            c0 = time.perf_counter()
            f.push_batch_raw(arr, nd, st)
            if sync_each:
                torch.cuda.synchronize()
                hlat.append((time.perf_counter() - c0) * 1e3)
        torch.cuda.synchronize()
        return time.perf_counter() - t0, hlat

    run_host(False)
    el_host, _ = run_host(False)
    _, hlat = run_host(True)
    f.status()
    assert torch.equal(hk, keep[:, :E].cpu()), "end-to-end keep codes differ from the device-resident run"
    bytes_h2d = S * E * W * H * 3
    e2e = {"frames_per_s": S * E / el_host, "latency_ms_p50": _pct(hlat, 50), "latency_ms_p99": _pct(hlat, 99),
           "calls": len(hplan), "h2d_bytes_per_call": bytes_h2d / len(hplan),
           "d2h_bytes_per_call": S * E * 5 / len(hplan), "h2d_gbs": bytes_h2d / el_host / 1e9,
           "how": f"the first {E} frames of every stream: pinned host frames in, pinned host scores and keep codes "
                  "out, through the same batched call"}
    del host_fr
    line = {"workload": f"serving: 32 streams x {T} uint8 RGB frames of 640x360, U{{1..8}} frames per stream per "
                        "batched call, B=32, L_max=30, tau_h=0.30",
            "calls": len(plan), "frames": frames_total,
            "pipelined_frames_per_s": frames_total / el_pipe, "pipelined_ms_per_call": el_pipe / len(plan) * 1e3,
            "graph_frames_per_s": frames_total / el_graph, "graph_ms_per_call": el_graph / len(plan) * 1e3,
            "sync_frames_per_s": frames_total / el_sync,
            "latency_ms_p50": _pct(lat, 50), "latency_ms_p99": _pct(lat, 99), "latency_ms_max": max(lat),
            "latency": "host wall time of one push_batch call plus a device synchronise",
            "keep_ratio": float((keep != 0).float().mean().item()), "e2e": e2e, "parity": par}
    f.close()
    return line


def bench_medium(args):
    print(json.dumps(medium_figures(args)), flush=True)


def medium_figures(args):
    """600 frames of 448x448 pushed 8 at a time: per-push latency and frames/s,
    and the keep codes and scores of the pipelined run against the oracle."""
    import numpy as np
    import torch

    import oracle as O
    import synth
    from paper_2609_03675_gb300 import NGFF
    spec = synth.medium()
    frames_np = synth.generate(spec)
    dev = torch.from_numpy(frames_np).cuda()
    scores = torch.empty(spec.frames, dtype=torch.float32, device="cuda")
    keep = torch.empty(spec.frames, dtype=torch.uint8, device="cuda")
    f = NGFF(spec.width, spec.height)
    st = torch.cuda.current_stream().cuda_stream
    fb = spec.frame_bytes
    ptrs = [(dev.data_ptr() + i * fb, scores.data_ptr() + 4 * i, keep.data_ptr() + i) for i in range(0, spec.frames, 8)]

    def run(sync_each):
        f.reset()
        lat = []
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for fp, sp, kp in ptrs:
            c0 = time.perf_counter()
            f.push_raw(0, fp, 8, sp, kp, None, st)
            if sync_each:
                torch.cuda.synchronize()
                lat.append((time.perf_counter() - c0) * 1e3)
        torch.cuda.synchronize()
        return time.perf_counter() - t0, lat

    for _ in range(max(1, args.warmup)):
        run(False)
    el_pipe, _ = run(False)
    f.status()
    o = O.load()
    _, so, ko = o.run(frames_np, O.Params(spec.width, spec.height))
    idx = f.candidates(0)
    par = parity_block(0.30, scores.cpu().numpy(), keep.cpu().numpy(), so, ko, idx=idx.cpu().numpy(),
                       want_idx=o.candidates(ko, 4))
    el_sync, lat = run(True)
    f.status()
    el_graph = _graph_seconds(lambda: [f.push_raw(0, fp, 8, sp, kp) for fp, sp, kp in ptrs], f.reset)
    f.status()
    # latency of one push launched from a graph (one 8-frame input buffer the
    # chunks are copied into, outside the timing), with a synchronise each
    buf = torch.empty_like(dev[:8])
    sc1 = torch.empty(8, dtype=torch.float32, device="cuda")
    kp1 = torch.empty(8, dtype=torch.uint8, device="cuda")
    g1 = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(g1):
        f.push(buf, scores=sc1, keep=kp1)
    f.reset()
    glat = []
    for i in range(0, spec.frames, 8):
        buf.copy_(dev[i:i + 8])
        torch.cuda.synchronize()
        c0 = time.perf_counter()
        g1.replay()
        torch.cuda.synchronize()
        glat.append((time.perf_counter() - c0) * 1e3)
    f.status()
    prof = f.profile_read()
    # end to end: the same pushes from pinned host frames, scores and keep
    # codes to pinned host memory, one synchronise at the end (and per push
    # for the latency), through the same C entry point
    host = torch.from_numpy(frames_np).pin_memory()
    hs = torch.empty(spec.frames, dtype=torch.float32, pin_memory=True)
    hk = torch.empty(spec.frames, dtype=torch.uint8, pin_memory=True)
    hptrs = [(host.data_ptr() + i * fb, hs.data_ptr() + 4 * i, hk.data_ptr() + i) for i in range(0, spec.frames, 8)]

    def run_host(sync_each):
        f.reset()
        lat = []
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for fp, sp, kp in hptrs:
            c0 = time.perf_counter()
            f.push_raw(0, fp, 8, sp, kp, None, st)
            if sync_each:
                torch.cuda.synchronize()
                lat.append((time.perf_counter() - c0) * 1e3)
        torch.cuda.synchronize()
        return time.perf_counter() - t0, lat

    run_host(False)
    el_host, _ = run_host(False)
    _, hlat = run_host(True)
    f.status()
    assert torch.equal(hk, keep.cpu()), "end-to-end keep codes differ from the device-resident run"
    f.close()
    return {"workload": "medium: 600 uint8 RGB frames of 448x448 pushed in chunks of 8, B=32, L_max=30, tau_h=0.30",
            "pushes": len(lat), "pipelined_frames_per_s": spec.frames / el_pipe,
            "sync_frames_per_s": spec.frames / el_sync,
            "graph_frames_per_s": spec.frames / el_graph, "graph_ms_per_push": el_graph / len(ptrs) * 1e3,
            "graph_latency_ms_p50": _pct(glat, 50), "graph_latency_ms_p99": _pct(glat, 99),
            "latency_ms_p50": _pct(lat, 50), "latency_ms_p99": _pct(lat, 99),
            "latency": "host wall time of one push plus a device synchronise",
            "e2e": {"frames_per_s": spec.frames / el_host, "latency_ms_p50": _pct(hlat, 50),
                    "latency_ms_p99": _pct(hlat, 99), "h2d_bytes_per_push": 8 * fb, "d2h_bytes_per_push": 8 * 5,
                    "how": "pinned host frames in, pinned host scores and keep codes out, through the same call"},
            "kernels_per_push": (prof["hist_launches"] + prof["select_launches"]) / max(1, prof["hist_launches"]),
            "kept": int((keep != 0).sum().item()), "parity": par}


def bench_rare_event(args):
    print(json.dumps(rare_event_figures(args)), flush=True)


def rare_event_figures(args):
    """3600 frames of 1280x720 with 40 injected events: frames/s, keep ratio
    and event-frame recall across tau_h; every tau's keep codes and scores
    against the oracle (one histogram pass on all host cores, its selection
    per tau)."""
    import numpy as np
    import torch

    import oracle as O
    import synth
    from paper_2609_03675_gb300 import NGFF
    spec = synth.rare_event()
    host = torch.empty((spec.frames, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.cuda()
    o = O.load()
    hist_o = o.histograms_parallel(host.data_ptr(), spec.frames, O.Params(spec.width, spec.height))
    # end to end at tau_h = 0.30: the whole stream from pinned host memory, outputs to pinned host memory
    fe = NGFF(spec.width, spec.height)
    hs = torch.empty(spec.frames, dtype=torch.float32, pin_memory=True)
    hk = torch.empty(spec.frames, dtype=torch.uint8, pin_memory=True)
    e2e_s = []
    for i in range(4):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        fe.reset()
        fe.push(host, scores=hs, keep=hk)
        torch.cuda.synchronize()
        if i:
            e2e_s.append(time.perf_counter() - t0)
    fe.status()
    fe.close()
    hk_e2e = hk.clone()
    del host
    events = torch.from_numpy(synth.event_mask(spec).astype(bool)).cuda()
    starts = synth.event_mask(spec)
    out = {"workload": "rare-event: 3600 uint8 RGB frames of 1280x720, 40 events of 1-3 frames, one whole-stream "
                       "push per step, B=32, L_max=30", "taus": {}}
    for tau in (0.30, 0.15, 0.10, 0.05, 0.02):
        f = NGFF(spec.width, spec.height, tau=tau)
        scores = torch.empty(spec.frames, dtype=torch.float32, device="cuda")
        keep = torch.empty(spec.frames, dtype=torch.uint8, device="cuda")

        def step():
            f.reset()
            f.push(dev, scores=scores, keep=keep)

        for _ in range(3):
            step()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(20):
            step()
        e1.record()
        torch.cuda.synchronize()
        f.status()
        kept = keep != 0
        # per-event recall: an event counts as caught if any of its frames is kept
        runs = _event_runs(starts.astype(bool))
        kc = kept.cpu().numpy()
        caught = sum(1 for a, b in runs if kc[a:b].any())
        so, ko = o.select(hist_o, O.Params(spec.width, spec.height, tau=tau))
        par = parity_block(tau, scores.cpu().numpy(), keep.cpu().numpy(), so, ko)
        if tau == 0.30:
            keep30 = keep.cpu().numpy()
        out["taus"][str(tau)] = {"frames_per_s": 20 * spec.frames / (e0.elapsed_time(e1) / 1e3),
                                 "keep_ratio": float(kept.float().mean().item()),
                                 "event_frame_recall": float(kept[events].float().mean().item()),
                                 "event_recall": caught / max(1, len(runs)),
                                 "parity": {"keep_equal": par["keep_equal"],
                                            "max_rel_score_err": par["max_rel_score_err"],
                                            "band_frames": par["band_frames"]}}
        f.close()
    t30 = out["taus"]["0.3"]
    el = statistics.median(e2e_s)
    out["e2e"] = {"frames_per_s": spec.frames / el, "ms_per_push": el * 1e3,
                  "h2d_bytes_per_push": spec.frames * spec.frame_bytes, "d2h_bytes_per_push": spec.frames * 5,
                  "statistic": "median of 3 whole-stream pushes at tau_h 0.30",
                  "keep_equal_device_run": bool(np.array_equal(hk_e2e.numpy(), keep30))}
    out["frames_per_s"] = t30["frames_per_s"]
    out["pixel_gbs"] = t30["frames_per_s"] * spec.frame_bytes / 1e9
    out["events"] = len(_event_runs(starts.astype(bool)))
    return out


def bench_gather(args):
    """Closing the 1080p prefix: candidate set S_c, then the gather of S_c into
    one buffer. Bandwidth of the gather (bytes read + written) against the
    measured copy peak."""
    import torch

    import synth
    from paper_2609_03675_gb300 import NGFF
    spec = synth.hd1080()
    spec = spec.with_(frames=min(spec.frames, max(1, args.frames)))
    host = torch.empty((spec.frames, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.cuda()
    del host
    f = NGFF(spec.width, spec.height, max_frames_per_push=spec.frames)
    f.push(dev)
    idx = f.candidates(0)
    m = idx.numel()
    out = torch.empty((m, spec.height, spec.width, 3), dtype=torch.uint8, device="cuda")
    m_dev = torch.empty(1, dtype=torch.int32, device="cuda")
    idx_buf = torch.empty(spec.frames, dtype=torch.int32, device="cuda")
    from paper_2609_03675_gb300 import _abi
    st = torch.cuda.current_stream().cuda_stream
    for _ in range(3):
        f.gather(dev, idx, out=out)
    torch.cuda.synchronize()
    reps = 50
    e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
    e0.record()
    for _ in range(reps):
        f.candidates_raw(0, idx_buf.data_ptr(), spec.frames, m_dev.data_ptr(), st)
    e1.record()
    for _ in range(reps):
        f.gather(dev, idx, out=out)
    e2.record()
    torch.cuda.synchronize()
    f.status()
    del _abi
    peak, kind = peaks()
    g_ms = e1.elapsed_time(e2) / reps
    gbs = 2 * m * spec.frame_bytes / (g_ms / 1e3) / 1e9
    print(json.dumps({"workload": f"finalize + gather of the 1080p stream ({spec.frames} frames, {m} candidates)",
                      "candidates_us": e0.elapsed_time(e1) / reps * 1e3, "gather_ms": g_ms,
                      "gather_bytes": 2 * m * spec.frame_bytes, "gather_gbs": gbs, "peak_gbs": peak,
                      "frac": gbs / peak, "peak_kind": f"{kind} copy bandwidth (read + write)"}), flush=True)


def bench_pipeline(args):
    """The coarse-to-fine path of one 1080p prefix on the device, per step:
    NGFF over the 3600 frames (Sec. 3.2), the candidate set S_c, the gather
    of S_c into the encoder's input buffer, and QER over S_c (Sec. 3.3) on
    synthetic visual keys standing in for the encoder's output (the encoder
    and the LLM are not part of this library). Time per phase from CUDA events."""
    import numpy as np
    import torch

    import synth
    from paper_2609_03675_gb300 import NGFF, QER
    from synth import qer as SQ
    spec = synth.hd1080()
    spec = spec.with_(frames=min(spec.frames, max(1, args.frames)))
    host = torch.empty((spec.frames, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.cuda()
    del host
    f = NGFF(spec.width, spec.height, max_frames_per_push=spec.frames)
    scores = torch.empty(spec.frames, dtype=torch.float32, device="cuda")
    keep = torch.empty(spec.frames, dtype=torch.uint8, device="cuda")
    f.push(dev, scores=scores, keep=keep)
    m = f.candidates(0).numel()  # the same every step (the stream restarts)
    f.reset()
    qs = SQ.QerSpec(n_frames=m)
    q, k, _ = SQ.generate(qs)
    qd = torch.from_numpy(q.view(np.int16)).cuda()
    kd = torch.from_numpy(k.view(np.int16)).cuda()
    fq = QER(qs.n_text, qs.n_heads, qs.n_kv_heads, qs.head_dim, m, qs.tokens_per_frame, 0.3)
    idx = torch.empty(spec.frames, dtype=torch.int32, device="cuda")
    m_dev = torch.empty(1, dtype=torch.int32, device="cuda")
    out = torch.empty((m, spec.height, spec.width, 3), dtype=torch.uint8, device="cuda")
    w = torch.empty(m, dtype=torch.float32, device="cuda")
    sel = torch.empty(m, dtype=torch.int32, device="cuda")
    k_dev = torch.zeros(1, dtype=torch.int32, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
    steps = max(1, min(args.steps, 50))
    acc = np.zeros(4)

    def step(timed):
        f.reset()
        if timed:
            ev[0].record()
        f.push(dev, scores=scores, keep=keep)
        if timed:
            ev[1].record()
        f.candidates_raw(0, idx.data_ptr(), spec.frames, m_dev.data_ptr(), st)
        if timed:
            ev[2].record()
        f.gather(dev, idx[:m], out=out)
        if timed:
            ev[3].record()
        fq.run_async(qd, kd, w, sel, k_dev)
        if timed:
            ev[4].record()

    for _ in range(max(3, args.warmup)):
        step(False)
    torch.cuda.synchronize()
    for _ in range(steps):
        step(True)
        torch.cuda.synchronize()
        acc += [ev[i].elapsed_time(ev[i + 1]) for i in range(4)]
    f.status()
    fq.status()
    assert int(m_dev.item()) == m
    ms = acc / steps
    print(json.dumps({
        "workload": f"pipeline: 1080p prefix of {spec.frames} frames -> NGFF -> S_c -> gather -> QER "
                    f"({qs.n_text} text tokens, {qs.tokens_per_frame} synthetic keys per frame)",
        "steps": steps, "ms_per_step": float(ms.sum()), "frames_per_s": spec.frames / (ms.sum() / 1e3),
        "candidates": m, "qer_selected": int(k_dev.item()),
        "drop_ratios": drop_ratios(spec.frames, m, int(k_dev.item())),
        "phase_ms": {"ngff_push": ms[0], "candidates": ms[1], "gather": ms[2], "qer": ms[3]},
        "timing": "CUDA events between phases on one stream, device synchronised after each step"}), flush=True)


def drop_ratios(frames: int, candidates: int, selected: int) -> dict:
    """Drop ratios of the coarse-to-fine path (Eq. 9): NGFF keeps `candidates`
    of `frames`, QER keeps `selected` of the candidates, and the total drop is
    D_total = 1 - (1 - D_NGFF)(1 - D_QER)."""
    d_ngff = 1.0 - candidates / frames if frames else 0.0
    d_qer = 1.0 - selected / candidates if candidates else 0.0
    return {"ngff": d_ngff, "qer": d_qer, "total": 1.0 - (1.0 - d_ngff) * (1.0 - d_qer)}


def peaks_bf16():
    try:
        with open(os.path.join(REPO, "MEASURED_PEAKS.json")) as fh:
            d = json.load(fh)
        return float(d["bf16_tflops"]), "measured"
    except Exception:  # noqa: BLE001
        return 1900.0, "fallback"


def bench_qer(args):
    """QER frame scoring (Eqs. 6-8) on the Qwen3-VL-8B last-layer geometry:
    256 text tokens, 32 query / 8 key heads of 128, 256 tokens per frame.
    Roofline of the tensor-core scoring kernel against both the measured
    bf16 dense peak and the measured copy bandwidth."""
    import numpy as np
    import torch

    from paper_2609_03675_gb300 import QER
    from synth import qer as SQ
    spec = SQ.QerSpec(n_frames=args.qer_frames)
    q, k, ev = SQ.generate(spec)
    qd = torch.from_numpy(q.view(np.int16)).cuda()
    kd = torch.from_numpy(k.view(np.int16)).cuda()
    f = QER(spec.n_text, spec.n_heads, spec.n_kv_heads, spec.head_dim, spec.n_frames, spec.tokens_per_frame, 0.3,
            kernel=args.qer_kernel)
    w = torch.empty(spec.n_frames, dtype=torch.float32, device="cuda")
    sel_all = torch.empty(spec.n_frames, dtype=torch.int32, device="cuda")
    k_dev = torch.zeros(1, dtype=torch.int32, device="cuda")
    for _ in range(5):
        f.run_async(qd, kd, w, sel_all, k_dev)
    torch.cuda.synchronize()
    reps = 200
    # the whole call, back to back (keys above L2: nothing stays cached between calls)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        f.run_async(qd, kd, w, sel_all, k_dev)
    e1.record()
    torch.cuda.synchronize()
    # the same call captured once into a CUDA graph, its launches back to back
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        f.run_async(qd, kd, w, sel_all, k_dev)
    for _ in range(3):
        g.replay()
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0.record()
    for _ in range(reps):
        g.replay()
    g1.record()
    torch.cuda.synchronize()
    # the scoring kernel alone, bracketed by events on the launching stream
    # (which also serialise it against the kernel before it)
    f.profile_reset(time_kernels=True)
    for _ in range(reps):
        f.run_async(qd, kd, w, sel_all, k_dev)
    torch.cuda.synchronize()
    f.status()
    sel = sel_all[: int(k_dev.item())]
    pr = f.profile_read()
    k_ms = pr["score_ms"] / max(pr["timed"], 1)
    tflops = pr["flops"] / pr["launches"] / (k_ms / 1e3) / 1e12
    gbs = pr["key_bytes"] / pr["launches"] / (k_ms / 1e3) / 1e9
    tc_peak, tc_kind = peaks_bf16()
    hbm_peak, hbm_kind = peaks()
    print(json.dumps({
        "workload": f"qer: {spec.n_text} text tokens, {spec.n_frames} frames x {spec.tokens_per_frame} tokens, "
                    f"{spec.n_heads}/{spec.n_kv_heads} heads of {spec.head_dim}, rho 0.3",
        "call_us": e0.elapsed_time(e1) / reps * 1e3, "score_kernel_us": k_ms * 1e3,
        "frames_per_s": spec.n_frames / (e0.elapsed_time(e1) / reps / 1e3),
        "graph_call_us": g0.elapsed_time(g1) / reps * 1e3,
        "tensor": {"achieved": tflops, "peak": tc_peak, "unit": "TFLOP/s", "frac": tflops / tc_peak,
                   "peak_kind": f"{tc_kind} bf16 dense (burst)",
                   "flops_per_launch": pr["flops"] / pr["launches"]},
        "hbm": {"achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak,
                "peak_kind": f"{hbm_kind} copy bandwidth", "key_bytes_per_launch": pr["key_bytes"] / pr["launches"]},
        "kernel_request": {0: "automatic", 1: "one-SM", 2: "paired-SM"}[args.qer_kernel],
        "selected": int(sel.numel()), "evidence_recovered": int(np.isin(ev, sel.cpu().numpy()).sum()),
        "n_evidence": int(len(ev))}), flush=True)


def bench_shards_ranks(args):
    """One 1080p stream split over the ranks of a torchrun job (strong
    scaling): every rank generates and prepares its shard plus halo, the gap
    maps are all-gathered (NCCL), every rank commits its shard. The time of a
    step is the max over ranks; the value counts the stream's frames."""
    import torch
    import torch.distributed as dist

    import synth
    from paper_2609_03675_gb300 import NGFF, shards
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    spec = synth.hd1080().with_(frames=min(3600, args.frames))
    T = spec.frames
    a, b, halo = shards.shard_bounds(T, world, rank, 30)
    host = torch.empty((b - a + halo, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, a - halo, b, out=host.data_ptr())
    dev = host.cuda()
    f = NGFF(spec.width, spec.height, max_frames_per_push=b - a + halo)

    def step():
        f.reset()
        return shards.sharded_push(f, dev, T, rank, world)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    dist.barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize()
    el = max_over_ranks(time.perf_counter() - t0)
    dist.barrier()
    f.status()
    if rank == 0:
        print(json.dumps({"workload": f"shards over ranks: the {T}-frame 1080p stream split over {world} GPUs",
                          "n_gpus": world, "scaling": "strong", "steps": args.steps,
                          "frames_per_s": T * args.steps / el, "ms_per_step": el / args.steps * 1e3,
                          "exchange": "one all-gather of the 30-entry gap maps per step (NCCL)",
                          "timing": "host wall time, max over ranks, device synchronised"}), flush=True)
    dist.destroy_process_group()


def bench_shards(args):
    """One 1080p stream split into 4 shards: each prepared from its frames and
    an L_max-frame halo (independently; on several GPUs they would run in
    parallel), chained through the gap maps, and committed. Reports the cost
    against one whole-stream push, and the checkpoint size and latency.
    Under torchrun (several ranks) the shards run one per GPU instead."""
    import torch

    import synth
    from paper_2609_03675_gb300 import NGFF
    if dist_env()[1] > 1:
        bench_shards_ranks(args)
        return
    spec = synth.hd1080().with_(frames=min(3600, args.frames))
    T = spec.frames
    host = torch.empty((T, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.cuda()
    del host
    S = 4
    bounds = [T * i // S for i in range(S + 1)]
    handles = [NGFF(spec.width, spec.height, max_frames_per_push=T) for _ in range(S)]
    single = NGFF(spec.width, spec.height, max_frames_per_push=T)
    keep_single = torch.empty(T, dtype=torch.uint8, device="cuda")

    def run_single():
        single.reset()
        _, k = single.push(dev, keep=keep_single)

    def run_sharded():
        maps, prep_ev = [], []
        for i in range(S):
            a, b = bounds[i], bounds[i + 1]
            halo = min(a, 30)
            maps.append(handles[i].shard_prepare(dev[a - halo:b], n_halo=halo, t0=a))
        g, keeps = 1, []
        for i in range(S):
            _, k = handles[i].shard_commit(g, bounds[i + 1] - bounds[i])
            keeps.append(k)
            g = int(maps[i][g - 1])
        return torch.cat(keeps)

    for _ in range(3):
        run_single()
        ks = run_sharded()
    torch.cuda.synchronize()
    assert torch.equal(ks, keep_single), "sharded decisions differ from the single pass"
    reps = 10
    t0 = time.perf_counter()
    for _ in range(reps):
        run_single()
    torch.cuda.synchronize()
    t_single = (time.perf_counter() - t0) / reps
    t0 = time.perf_counter()
    for _ in range(reps):
        run_sharded()
    torch.cuda.synchronize()
    t_sharded = (time.perf_counter() - t0) / reps
    # checkpoint / resume of one stream
    state = single.state_save()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(100):
        single.state_save(out=state)
    t_save = (time.perf_counter() - t0) / 100
    t0 = time.perf_counter()
    for _ in range(100):
        single.state_load(state)
    t_load = (time.perf_counter() - t0) / 100
    print(json.dumps({
        "workload": f"shards: the {T}-frame 1080p stream in {S} shards, prepared and committed on one GPU",
        "single_push_ms": t_single * 1e3, "sharded_ms": t_sharded * 1e3,
        "sharded_over_single": t_sharded / t_single,
        "halo_frames_extra": sum(min(bounds[i], 30) for i in range(S)),
        "decisions_equal": True,
        "state_bytes": int(state.numel()), "state_save_us": t_save * 1e6, "state_load_us": t_load * 1e6,
        "timing": "host wall time with a device synchronise around each batch of repetitions"}), flush=True)


def bench_signals(args):
    """The NGFF signals on the 1080p stream (frames/s, first-stage
    bandwidth against the measured copy peak) and on the 720p rare-event
    stream (keep ratio and event recall across thresholds): the synthetic
    counterpart of the paper's signal ablation."""
    import torch

    import synth
    from paper_2609_03675_gb300 import NGFF
    names = {0: "histogram", 1: "lowres", 2: "dhash", 3: "scd"}
    taus = {0: (0.30, 0.10, 0.05), 1: (0.05, 0.02, 0.01), 2: (0.20, 0.10, 0.05), 3: (0.30, 0.10, 0.05)}
    peak, peak_kind = peaks()
    spec = synth.hd1080()
    T = min(spec.frames, 600)
    spec = spec.with_(frames=T)
    host = torch.empty((T, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(spec, out=host.data_ptr())
    dev = host.cuda()
    scores = torch.empty(T, dtype=torch.float32, device="cuda")
    keep = torch.empty(T, dtype=torch.uint8, device="cuda")
    out = {"workload": f"signals: 1080p stream of {T} frames (throughput), 720p rare-event stream of 3600 frames "
                       "with 40 events (recall)", "peak_gbs": peak, "peak_kind": f"{peak_kind} copy bandwidth",
           "signals": {}}
    for sig, name in names.items():
        f = NGFF(spec.width, spec.height, max_frames_per_push=T, signal=sig)

        def step():
            f.reset()
            f.push(dev, scores=scores, keep=keep)

        for _ in range(max(3, args.warmup)):
            step()
        torch.cuda.synchronize()
        f.profile_reset(time_kernels=True)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(20):
            step()
        e1.record()
        torch.cuda.synchronize()
        f.status()
        prof = f.profile_read()
        ms = e0.elapsed_time(e1) / 20
        k_ms = prof["hist_ms"] / max(prof["hist_timed"], 1)
        k_bytes = prof["hist_bytes"] / max(prof["hist_launches"], 1)
        out["signals"][name] = {"frames_per_s": T / (ms / 1e3), "ms_per_step": ms, "first_stage_ms": k_ms,
                                "first_stage_gbs": k_bytes / (k_ms / 1e3) / 1e9,
                                "first_stage_frac": k_bytes / (k_ms / 1e3) / 1e9 / peak,
                                "select_ms": prof["select_ms"] / max(prof["select_timed"], 1),
                                "keep_ratio_default_tau": float((keep != 0).float().mean().item())}
        f.close()
    del dev, host
    rs = synth.rare_event()
    rhost = torch.empty((rs.frames, rs.height, rs.width, 3), dtype=torch.uint8, pin_memory=True)
    synth.generate(rs, out=rhost.data_ptr())
    rdev = rhost.cuda()
    ev = synth.event_mask(rs).astype(bool)
    runs, t = [], 0
    while t < rs.frames:
        if ev[t]:
            u = t
            while u < rs.frames and ev[u]:
                u += 1
            runs.append((t, u))
            t = u
        else:
            t += 1
    rk = torch.empty(rs.frames, dtype=torch.uint8, device="cuda")
    rsc = torch.empty(rs.frames, dtype=torch.float32, device="cuda")
    for sig, name in names.items():
        rec = {}
        for tau in taus[sig]:
            f = NGFF(rs.width, rs.height, tau=tau, signal=sig)
            f.push(rdev, scores=rsc, keep=rk)
            torch.cuda.synchronize()
            f.status()
            kc = rk.cpu().numpy() != 0
            rec[str(tau)] = {"keep_ratio": float(kc.mean()), "event_frame_recall": float(kc[ev].mean()),
                             "event_recall": sum(1 for a, b in runs if kc[a:b].any()) / max(1, len(runs))}
            f.close()
        out["signals"][name]["rare_event"] = rec
    print(json.dumps(out), flush=True)


SENSITIVITY_ROWS = (  # (M_min, L_max, tau_h): the rows of the paper's NGFF sensitivity table (App. B.2)
    (2, 30, 0.30), (4, 30, 0.30), (8, 30, 0.30),
    (4, 15, 0.30), (4, 45, 0.30),
    (4, 30, 0.15), (4, 30, 0.45), (4, 30, 0.60), (4, 30, 0.75))


def bench_sensitivity(args):
    """The synthetic counterpart of the paper's NGFF sensitivity table: for
    each (M_min, L_max, tau_h) row, the stream is pushed whole and closed, and
    the line reports the drop ratio 1 - |S_c| / T (the last frame and the
    M_min fill included), the device-resident frames/s of push + close, and
    the keep codes and candidate set against the oracle. Streams: the 1080p
    stream (3600 frames; its scene cuts change the histogram by far more than
    any tau of the table and little else moves it), the medium stream (600
    frames with brightness drift, pushed whole) and the tiny stream (64
    frames, where M_min can matter)."""
    import numpy as np
    import torch

    import oracle as O
    import synth
    from paper_2609_03675_gb300 import NGFF
    out = {"workload": "sensitivity: the rows of the NGFF sensitivity table on the 1080p, medium and tiny streams",
           "fields": ["m_min", "l_max", "tau", "drop_pct", "frames_per_s", "keep_equal", "candidates_equal"],
           "streams": {}}
    o = O.load()
    for name, spec in (("1080p", synth.hd1080()), ("medium", synth.medium()), ("tiny", synth.tiny())):
        T = spec.frames
        host = torch.empty((T, spec.height, spec.width, 3), dtype=torch.uint8, pin_memory=True)
        synth.generate(spec, out=host.data_ptr())
        dev = host.cuda()
        hist_o = o.histograms_parallel(host.data_ptr(), T, O.Params(spec.width, spec.height))
        del host
        keep = torch.empty(T, dtype=torch.uint8, device="cuda")
        idx = torch.empty(T, dtype=torch.int32, device="cuda")
        m_dev = torch.zeros(1, dtype=torch.int32, device="cuda")
        rows = []
        for m_min, l_max, tau in SENSITIVITY_ROWS:
            f = NGFF(spec.width, spec.height, m_min=m_min, l_max=l_max, tau=tau, max_frames_per_push=T)

            def step():
                f.reset()
                f.push(dev, keep=keep)
                f.candidates_raw(0, idx.data_ptr(), T, m_dev.data_ptr())

            for _ in range(3):
                step()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            reps = 10
            e0.record()
            for _ in range(reps):
                step()
            e1.record()
            torch.cuda.synchronize()
            f.status()
            m = int(m_dev.item())
            _, ko = o.select(hist_o, O.Params(spec.width, spec.height, m_min=m_min, l_max=l_max, tau=tau))
            want = o.candidates(ko, m_min)
            rows.append([m_min, l_max, tau, round(100.0 * (1.0 - m / T), 2),
                         round(reps * T / (e0.elapsed_time(e1) / 1e3)),
                         bool(np.array_equal(keep.cpu().numpy(), ko)),
                         bool(np.array_equal(idx[:m].cpu().numpy().astype(np.uint32), want))])
            f.close()
        out["streams"][name] = {"frames": T, "size": f"{spec.width}x{spec.height}", "rows": rows}
        del dev
        torch.cuda.empty_cache()
    print(json.dumps(out), flush=True)


def bench_static(args):
    """cofie_ngff_select_static (the allocation-free selection) at
    the largest sizes its static array admits and at a typical one: CUDA
    events around repeated calls on histograms already on the device."""
    import ctypes

    import numpy as np
    import torch

    from paper_2609_03675_gb300 import _abi
    lib = _abi.load()
    st = torch.cuda.current_stream().cuda_stream
    out = {"workload": "cofie_ngff_select_static: decisions of a fresh stream from its histograms (a grid of "
                       "distance warps, then one scan CTA)",
           "cases": []}
    g = np.random.default_rng(7)
    for n, bins, l_max in ((3600, 32, 30), (33825, 32, 30), (3970, 256, 256)):
        hist = torch.from_numpy(g.integers(0, 4096, size=(n, bins), dtype=np.int32)).cuda()
        s = torch.empty(n, dtype=torch.float32, device="cuda")
        k = torch.empty(n, dtype=torch.uint8, device="cuda")
        p = _abi.Params()
        lib.cofie_ngff_default_params(ctypes.byref(p), 1920, 1080)
        p.bins, p.l_max, p.tau = bins, l_max, 0.3
        err = ctypes.create_string_buffer(256)

        def call():
            rc = lib.cofie_ngff_select_static(ctypes.byref(p), hist.data_ptr(), n, s.data_ptr(), k.data_ptr(), err,
                                              len(err), st)
            assert rc == 0, err.value

        for _ in range(3):
            call()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = 10
        e0.record()
        for _ in range(reps):
            call()
        e1.record()
        torch.cuda.synchronize()
        out["cases"].append({"frames": n, "bins": bins, "l_max": l_max, "ms_per_call": e0.elapsed_time(e1) / reps,
                             "scratch_words": n * (l_max + (l_max + 31) // 32)})
    print(json.dumps(out), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        bench_reference(args)
    elif args.workload == "serving":
        bench_serving(args)
    elif args.workload == "medium":
        bench_medium(args)
    elif args.workload == "pipeline":
        bench_pipeline(args)
    elif args.workload == "rare_event":
        bench_rare_event(args)
    elif args.workload == "gather":
        bench_gather(args)
    elif args.workload == "qer":
        bench_qer(args)
    elif args.workload == "shards":
        bench_shards(args)
    elif args.workload == "signals":
        bench_signals(args)
    elif args.workload == "tiny":
        print(json.dumps(tiny_figures(args)), flush=True)
    elif args.workload == "static":
        bench_static(args)
    elif args.workload == "sensitivity":
        bench_sensitivity(args)
    else:
        bench_gb300(args)


if __name__ == "__main__":
    main()
