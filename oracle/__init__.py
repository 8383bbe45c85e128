"""ORACLE for NGFF (CoFiE Sec. 3.2) -- test infrastructure only.

A plain, slow, single-threaded C restatement of the method
(``ngff_oracle.c``), built with the host C compiler on first use and loaded
with ctypes. Only the tests, ``__graft_entry__.smoke()`` and the benchmark's
CPU-baseline leg may import this package. The GPU library never calls it and
shares no code, header or table with it.

Functions mirror the C entry points:
  luma, luma_map, bin_of -- steps 1-2 on single values / pixel arrays
  histogram             -- step 2 on one frame
  tv                    -- Eq. 2 (double), tv32 the fp32 decision value
  select                -- Eqs. 3-5 on given histograms
  run                   -- steps 1-5 over a stream
  candidates            -- the safeguards that close a prefix (last frame,
                           M_min uniform fill)
  histograms_parallel   -- the oracle's own histogram routine mapped over
                           frames on several host threads (ctypes releases the
                           GIL), for full-size streams
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ngff_oracle.c")
_LIB = os.path.join(_HERE, "libngff_oracle.so")
_lock = threading.Lock()
_lib = None

KEEP_DROP, KEEP_NOVELTY, KEEP_GAP, KEEP_FIRST = 0, 1, 2, 3


class _Params(ctypes.Structure):
    _fields_ = [
        ("width", ctypes.c_uint32),
        ("height", ctypes.c_uint32),
        ("bins", ctypes.c_uint32),
        ("l_max", ctypes.c_uint32),
        ("m_min", ctypes.c_uint32),
        ("tau", ctypes.c_float),
        ("luma_w", ctypes.c_uint32 * 3),
        ("luma_den", ctypes.c_uint32),
    ]


@dataclass(frozen=True)
class Params:
    """NGFF hyperparameters; defaults B=32 (App. A), M_min=4, L_max=30, tau_h=0.30
    (the configuration held fixed in the sensitivity study, App. B.2)."""
    width: int
    height: int
    bins: int = 32
    l_max: int = 30
    m_min: int = 4
    tau: float = 0.30
    luma_w: tuple = (299, 587, 114)
    luma_den: int = 1000

    @property
    def npix(self) -> int:
        return self.width * self.height

    def _c(self) -> _Params:
        return _Params(self.width, self.height, self.bins, self.l_max, self.m_min, self.tau,
                       (ctypes.c_uint32 * 3)(*self.luma_w), self.luma_den)


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle C file into a shared library (idempotent)."""
    with _lock:
        stale = (not os.path.exists(out)) or os.path.getmtime(out) < os.path.getmtime(src)
        if force or stale:
            tmp = out + f".tmp{os.getpid()}"
            subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-ffp-contract=off",
                            "-Wall", "-o", tmp, src], check=True)
            os.replace(tmp, out)
    return out


def _bind(lib):
    P = ctypes.POINTER(_Params)
    vp = ctypes.c_void_p
    lib.ngff_oracle_luma.argtypes = [ctypes.c_uint32] * 3 + [P]
    lib.ngff_oracle_luma.restype = ctypes.c_uint32
    lib.ngff_oracle_luma_map.argtypes = [vp, ctypes.c_uint64, P, vp]
    lib.ngff_oracle_luma_map.restype = None
    lib.ngff_oracle_bin.argtypes = [ctypes.c_uint32, ctypes.c_uint32]
    lib.ngff_oracle_bin.restype = ctypes.c_uint32
    lib.ngff_oracle_histogram.argtypes = [vp, P, vp]
    lib.ngff_oracle_histogram.restype = None
    lib.ngff_oracle_tv.argtypes = [vp, vp, ctypes.c_uint32, ctypes.c_uint64]
    lib.ngff_oracle_tv.restype = ctypes.c_double
    lib.ngff_oracle_tv32.argtypes = [vp, vp, ctypes.c_uint32, ctypes.c_uint64]
    lib.ngff_oracle_tv32.restype = ctypes.c_float
    lib.ngff_oracle_select.argtypes = [vp, ctypes.c_uint32, P, vp, vp]
    lib.ngff_oracle_select.restype = ctypes.c_int
    lib.ngff_oracle_run.argtypes = [vp, ctypes.c_uint32, P, vp, vp, vp]
    lib.ngff_oracle_run.restype = ctypes.c_int
    lib.ngff_oracle_candidates.argtypes = [vp, ctypes.c_uint32, ctypes.c_uint32, vp, vp]
    lib.ngff_oracle_candidates.restype = ctypes.c_int
    return lib


class Oracle:
    """One loaded copy of the oracle library (the default, or a test variant)."""

    def __init__(self, path: str):
        self.path = path
        self.lib = _bind(ctypes.CDLL(path))

    def luma(self, r, g, b, p: Params) -> int:
        c = p._c()
        return int(self.lib.ngff_oracle_luma(int(r), int(g), int(b), ctypes.byref(c)))

    def luma_map(self, pixels: np.ndarray, p: Params) -> np.ndarray:
        """Intensity of every RGB triple in ``pixels`` (uint8 [..., 3])."""
        px = np.ascontiguousarray(pixels, dtype=np.uint8)
        n = px.size // 3
        out = np.zeros(n, dtype=np.uint8)
        c = p._c()
        self.lib.ngff_oracle_luma_map(px.ctypes.data, n, ctypes.byref(c), out.ctypes.data)
        return out.reshape(px.shape[:-1])

    def bin_of(self, y: int, bins: int) -> int:
        return int(self.lib.ngff_oracle_bin(int(y), int(bins)))

    def histogram(self, frame: np.ndarray, p: Params) -> np.ndarray:
        f = np.ascontiguousarray(frame, dtype=np.uint8)
        assert f.size == 3 * p.npix
        out = np.zeros(p.bins, dtype=np.uint32)
        c = p._c()
        self.lib.ngff_oracle_histogram(f.ctypes.data, ctypes.byref(c), out.ctypes.data)
        return out

    def tv(self, ci, cj, npix: int) -> float:
        a = np.ascontiguousarray(ci, dtype=np.uint32)
        b = np.ascontiguousarray(cj, dtype=np.uint32)
        return float(self.lib.ngff_oracle_tv(a.ctypes.data, b.ctypes.data, a.size, npix))

    def tv32(self, ci, cj, npix: int) -> float:
        a = np.ascontiguousarray(ci, dtype=np.uint32)
        b = np.ascontiguousarray(cj, dtype=np.uint32)
        return float(self.lib.ngff_oracle_tv32(a.ctypes.data, b.ctypes.data, a.size, npix))

    def select(self, hist: np.ndarray, p: Params):
        h = np.ascontiguousarray(hist, dtype=np.uint32)
        T = h.shape[0]
        score = np.zeros(T, dtype=np.float64)
        keep = np.zeros(T, dtype=np.uint8)
        c = p._c()
        rc = self.lib.ngff_oracle_select(h.ctypes.data, T, ctypes.byref(c), score.ctypes.data, keep.ctypes.data)
        if rc != 0:
            raise ValueError(f"ngff_oracle_select failed ({rc})")
        return score, keep

    def run(self, frames: np.ndarray, p: Params):
        f = np.ascontiguousarray(frames, dtype=np.uint8)
        T = f.shape[0]
        hist = np.zeros((T, p.bins), dtype=np.uint32)
        score = np.zeros(T, dtype=np.float64)
        keep = np.zeros(T, dtype=np.uint8)
        c = p._c()
        rc = self.lib.ngff_oracle_run(f.ctypes.data, T, ctypes.byref(c), hist.ctypes.data,
                                      score.ctypes.data, keep.ctypes.data)
        if rc != 0:
            raise ValueError(f"ngff_oracle_run failed ({rc})")
        return hist, score, keep

    def candidates(self, keep: np.ndarray, m_min: int) -> np.ndarray:
        k = np.ascontiguousarray(keep, dtype=np.uint8)
        T = k.size
        idx = np.zeros(max(T, 1), dtype=np.uint32)
        m = ctypes.c_uint32(0)
        rc = self.lib.ngff_oracle_candidates(k.ctypes.data, T, m_min, idx.ctypes.data, ctypes.byref(m))
        if rc != 0:
            raise ValueError(f"ngff_oracle_candidates failed ({rc})")
        return idx[: m.value].copy()

    def histograms_parallel(self, frames_ptr: int, T: int, p: Params, nthreads: int | None = None,
                            frame_ids=None) -> np.ndarray:
        """The oracle's histogram routine on frames at host address ``frames_ptr``
        (T frames back to back), mapped over threads. ``frame_ids`` restricts it
        to a subset (rows follow ``frame_ids``)."""
        ids = np.arange(T) if frame_ids is None else np.asarray(frame_ids)
        out = np.zeros((len(ids), p.bins), dtype=np.uint32)
        fb = 3 * p.npix
        c = p._c()
        nthreads = nthreads or max(1, len(os.sched_getaffinity(0)))

        def work(j):
            self.lib.ngff_oracle_histogram(ctypes.c_void_p(frames_ptr + int(ids[j]) * fb), ctypes.byref(c),
                                           ctypes.c_void_p(out[j].ctypes.data))

        with ThreadPoolExecutor(max_workers=nthreads) as ex:
            list(ex.map(work, range(len(ids))))
        return out


_default = None


def load() -> Oracle:
    """The oracle built from ngff_oracle.c."""
    global _default
    if _default is None:
        _default = Oracle(build())
    return _default
