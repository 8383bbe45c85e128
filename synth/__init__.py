"""Seeded synthetic RGB video streams for the tests and the benchmark.

Input generation only: this package holds none of the filtering method's
arithmetic. Both the oracle and the GPU path consume the bytes it writes.
The C core (``framegen.c``) is built on first use with the host compiler and
is integer-only, so a seed gives identical frames on x86_64 and aarch64.

The five stream recipes below stand in for the paper's benchmark videos
(StreamingBench, OvO-Bench and the offline suites), which state no frame size
or sampling rate; sizes and scene statistics follow the workload definitions
of the filtering benchmark (tiny 224x224, medium 448x448, 1080p, 32-stream
640x360 serving, 720p rare-event).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "framegen.c")
_LIB = os.path.join(_HERE, "libframegen.so")
_lock = threading.Lock()
_lib = None

UNIFORM_SCENES = 1
GRADIENT_DRIFT = 2
TEXTURE_WALK = 3
BANDED_SCENES = 4


class _Spec(ctypes.Structure):
    _fields_ = [
        ("recipe", ctypes.c_int32),
        ("width", ctypes.c_uint32),
        ("height", ctypes.c_uint32),
        ("frames", ctypes.c_uint32),
        ("seed", ctypes.c_uint64),
        ("sigma", ctypes.c_uint32),
        ("scene_len", ctypes.c_uint32),
        ("mean_scene_len", ctypes.c_uint32),
        ("n_events", ctypes.c_uint32),
    ]


def build(force: bool = False) -> str:
    """Compile framegen.c into libframegen.so next to it (idempotent)."""
    with _lock:
        stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
        if force or stale:
            tmp = _LIB + f".tmp{os.getpid()}"
            subprocess.run(
                ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-ffp-contract=off",
                 "-pthread", "-Wall", "-o", tmp, _SRC],
                check=True,
            )
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        lib.synth_generate.argtypes = [ctypes.POINTER(_Spec), ctypes.c_uint32, ctypes.c_uint32,
                                       ctypes.c_void_p, ctypes.c_int]
        lib.synth_generate.restype = ctypes.c_int
        lib.synth_scene_starts.argtypes = [ctypes.POINTER(_Spec), ctypes.c_void_p, ctypes.c_uint32,
                                           ctypes.POINTER(ctypes.c_uint32)]
        lib.synth_scene_starts.restype = ctypes.c_int
        lib.synth_event_frames.argtypes = [ctypes.POINTER(_Spec), ctypes.c_void_p]
        lib.synth_event_frames.restype = ctypes.c_int
        lib.synth_u64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.synth_u64.restype = ctypes.c_uint64
        _lib = lib
    return _lib


@dataclass(frozen=True)
class StreamSpec:
    recipe: int
    width: int
    height: int
    frames: int
    seed: int
    sigma: int = 0
    scene_len: int = 0
    mean_scene_len: int = 0
    n_events: int = 0

    @property
    def frame_bytes(self) -> int:
        return 3 * self.width * self.height

    @property
    def total_bytes(self) -> int:
        return self.frames * self.frame_bytes

    def with_(self, **kw) -> "StreamSpec":
        d = self.__dict__.copy()
        d.update(kw)
        return StreamSpec(**d)

    def _c(self) -> _Spec:
        return _Spec(self.recipe, self.width, self.height, self.frames, self.seed & (2**64 - 1),
                     self.sigma, self.scene_len, self.mean_scene_len, self.n_events)


SEED_BASE = 0xC0F1E000


def tiny(seed: int | None = None) -> StreamSpec:
    """64 frames of 224x224: 4 scenes x 16 frames, uniform-random bases, noise sigma 4."""
    return StreamSpec(UNIFORM_SCENES, 224, 224, 64, SEED_BASE + 1 if seed is None else seed,
                      sigma=4, scene_len=16)


def tiny_banded(seed: int | None = None) -> StreamSpec:
    """The tiny stream with scene s drawn from the band [64 s, 64 s + 63] per channel."""
    return StreamSpec(BANDED_SCENES, 224, 224, 64, SEED_BASE + 1 if seed is None else seed,
                      sigma=4, scene_len=16)


def medium(seed: int | None = None) -> StreamSpec:
    """600 frames of 448x448: geometric scenes (mean 20), gradients with +-1 drift, sigma 3."""
    return StreamSpec(GRADIENT_DRIFT, 448, 448, 600, SEED_BASE + 2 if seed is None else seed,
                      sigma=3, mean_scene_len=20)


def hd1080(seed: int | None = None) -> StreamSpec:
    """3600 frames of 1920x1080: geometric scenes (mean 150), translating textures, sigma 2."""
    return StreamSpec(TEXTURE_WALK, 1920, 1080, 3600, SEED_BASE + 3 if seed is None else seed,
                      sigma=2, mean_scene_len=150)


def serving_stream(stream: int, seed: int | None = None) -> StreamSpec:
    """One of the 32 serving streams: 1800 frames of 640x360, the medium recipe."""
    base = SEED_BASE + 4 if seed is None else seed
    return StreamSpec(GRADIENT_DRIFT, 640, 360, 1800, base + stream, sigma=3, mean_scene_len=20)


def rare_event(seed: int | None = None) -> StreamSpec:
    """3600 frames of 1280x720, the medium recipe, with 40 injected 1-3 frame events."""
    return StreamSpec(GRADIENT_DRIFT, 1280, 720, 3600, SEED_BASE + 5 if seed is None else seed,
                      sigma=3, mean_scene_len=20, n_events=40)


SERVING_STREAMS = 32


def generate(spec: StreamSpec, f0: int = 0, f1: int | None = None, out=None,
             nthreads: int | None = None) -> np.ndarray | None:
    """Frames [f0, f1) as uint8 [n, H, W, 3].

    ``out`` may be None (a new numpy array is returned), a writable numpy
    array, or an integer host address of at least n*H*W*3 bytes (for example
    a pinned torch tensor's ``data_ptr()``), in which case None is returned.
    """
    f1 = spec.frames if f1 is None else f1
    if not (0 <= f0 <= f1 <= spec.frames):
        raise ValueError("frame range out of bounds")
    n = f1 - f0
    if nthreads is None:
        nthreads = max(1, len(os.sched_getaffinity(0)))
    lib = _load()
    c = spec._c()
    ret = None
    if out is None:
        ret = np.empty((n, spec.height, spec.width, 3), dtype=np.uint8)
        ptr = ret.ctypes.data
    elif isinstance(out, np.ndarray):
        if out.dtype != np.uint8 or out.nbytes < n * spec.frame_bytes or not out.flags.c_contiguous:
            raise ValueError("out must be a contiguous uint8 array of the stream's size")
        ptr = out.ctypes.data
        ret = out
    else:
        ptr = int(out)
    if n and lib.synth_generate(ctypes.byref(c), f0, f1, ctypes.c_void_p(ptr), nthreads) != 0:
        raise RuntimeError("synth_generate failed")
    return ret if out is None or isinstance(out, np.ndarray) else None


def scene_starts(spec: StreamSpec) -> np.ndarray:
    """Index of the first frame of every scene (the ground-truth cuts are entries 1..)."""
    lib = _load()
    c = spec._c()
    cap = spec.frames + 1
    buf = np.empty(cap, dtype=np.uint32)
    cnt = ctypes.c_uint32(0)
    lib.synth_scene_starts(ctypes.byref(c), ctypes.c_void_p(buf.ctypes.data), cap, ctypes.byref(cnt))
    return buf[: cnt.value].copy()


def event_mask(spec: StreamSpec) -> np.ndarray:
    """uint8 [frames]: 1 where an injected event touches the frame."""
    lib = _load()
    c = spec._c()
    m = np.zeros(spec.frames, dtype=np.uint8)
    lib.synth_event_frames(ctypes.byref(c), ctypes.c_void_p(m.ctypes.data))
    return m


def u64(key: int, i: int) -> int:
    """The counter-based generator's i-th output for ``key`` (SplitMix64)."""
    return int(_load().synth_u64(key & (2**64 - 1), i))


def push_sizes(seed: int, stream: int, count: int, lo: int = 1, hi: int = 8) -> np.ndarray:
    """Per-call push sizes U{lo..hi} for one serving stream (multiply-shift of 32 bits)."""
    key = (seed * 0x100000001B3 + stream) & (2**64 - 1)
    span = hi - lo + 1
    return np.array([lo + (((u64(key, i) >> 32) * span) >> 32) for i in range(count)], dtype=np.int64)
