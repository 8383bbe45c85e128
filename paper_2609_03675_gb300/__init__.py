"""NGFF (CoFiE's Novelty-Guided Frame Filtering, Sec. 3.2) on GB300.

Thin Python binding of libcofie_ngff.so. Every step of the method runs in the
library's CUDA kernels; this module only marshals arguments. PyTorch provides
device memory and the current CUDA stream.

    from paper_2609_03675_gb300 import NGFF
    f = NGFF(1920, 1080)                 # B=32, L_max=30, M_min=4, tau_h=0.30
    scores, keep = f.push(frames_u8)     # frames: uint8 [n, H, W, 3], cuda or cpu
"""
from __future__ import annotations

import ctypes

import torch

from . import _abi
from ._abi import (KEEP_DROP, KEEP_FIRST, KEEP_GAP, KEEP_NOVELTY, NGFFError)  # noqa: F401

__all__ = ["NGFF", "QER", "NGFFError", "KEEP_DROP", "KEEP_NOVELTY", "KEEP_GAP", "KEEP_FIRST", "library_path"]


def library_path() -> str:
    return _abi.LIB_PATH


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, torch.Tensor):
        if not x.is_contiguous():
            raise ValueError("tensors passed to the library must be contiguous")
        return x.data_ptr()
    return int(x)


class NGFF:
    """One library handle: max_streams independent streams of width x height frames."""

    def __init__(self, width: int, height: int, *, bins: int = 32, l_max: int = 30, m_min: int = 4,
                 tau: float = 0.30, luma_weights=(299, 587, 114), luma_den: int = 1000, max_streams: int = 1,
                 max_frames_per_push: int = 4096, device: int | None = None, host_stage_bytes: int = 0,
                 signal: int = 0, scd_cut: float | None = None, scd_gradual: float | None = None,
                 max_stream_frames: int = 0):
        lib = _abi.load()
        p = _abi.Params()
        lib.cofie_ngff_default_params(ctypes.byref(p), width, height)
        p.bins, p.l_max, p.m_min, p.tau = bins, l_max, m_min, tau
        p.luma_w[0], p.luma_w[1], p.luma_w[2] = luma_weights
        p.luma_den = luma_den
        p.max_streams, p.max_frames_per_push = max_streams, max_frames_per_push
        if device is None:
            device = torch.cuda.current_device()
        p.device = device
        p.host_stage_bytes = host_stage_bytes
        p.signal = signal
        if scd_cut is not None:
            p.scd_cut = scd_cut
        if scd_gradual is not None:
            p.scd_gradual = scd_gradual
        p.max_stream_frames = max_stream_frames
        h = ctypes.c_void_p()
        rc = lib.cofie_ngff_create(ctypes.byref(p), ctypes.byref(h))
        if rc != _abi.OK:
            raise NGFFError(rc, lib.cofie_ngff_global_error().decode())
        self._lib, self._h, self.params = lib, h, p
        self.width, self.height, self.bins, self.l_max, self.m_min, self.tau = width, height, bins, l_max, m_min, tau
        self.device = torch.device("cuda", device)
        self.frame_bytes = 3 * width * height
        self.signal = signal
        self.feature_words = int(lib.cofie_ngff_feature_words(h))

    # ----------------------------------------------------------------- util --
    def _check(self, rc: int):
        if rc != _abi.OK:
            raise NGFFError(rc, self._lib.cofie_ngff_last_error(self._h).decode())

    def _stream(self, cuda_stream):
        if cuda_stream is None:
            return torch.cuda.current_stream(self.device).cuda_stream
        if isinstance(cuda_stream, torch.cuda.Stream):
            return cuda_stream.cuda_stream
        return int(cuda_stream)

    def _outputs(self, frames, n, scores, keep, hist, want_hist):
        on_gpu = isinstance(frames, torch.Tensor) and frames.is_cuda
        kw = dict(device=self.device) if on_gpu else dict(pin_memory=True)
        if scores is None:
            scores = torch.empty(n, dtype=torch.float32, **kw)
        if keep is None:
            keep = torch.empty(n, dtype=torch.uint8, **kw)
        if want_hist and hist is None:
            hist = torch.empty((n, self.feature_words), dtype=torch.int32, **kw)
        return scores, keep, hist

    def _frames(self, frames):
        if isinstance(frames, torch.Tensor):
            if frames.dtype != torch.uint8:
                raise ValueError("frames must be uint8")
            if frames.numel() % self.frame_bytes:
                raise ValueError("frames must hold whole width x height x 3 frames")
            return frames.numel() // self.frame_bytes
        raise TypeError("frames must be a torch.uint8 tensor [n, H, W, 3] (cuda or cpu)")

    # ------------------------------------------------------------------ API --
    def push(self, frames, stream: int = 0, *, scores=None, keep=None, hist=None, return_hist: bool = False,
             cuda_stream=None):
        """Decides the next n frames of ``stream``; returns (scores, keep) or
        (scores, keep, hist). Asynchronous on the current CUDA stream."""
        n = self._frames(frames)
        scores, keep, hist = self._outputs(frames, n, scores, keep, hist, return_hist or hist is not None)
        st = self._stream(cuda_stream)
        if hist is None:
            rc = self._lib.cofie_ngff_push(self._h, stream, _ptr(frames), n, _ptr(scores), _ptr(keep), st)
        else:
            rc = self._lib.cofie_ngff_push_ex(self._h, stream, _ptr(frames), n, _ptr(scores), _ptr(keep),
                                              _ptr(hist), st)
        self._check(rc)
        return (scores, keep, hist) if hist is not None else (scores, keep)

    def push_raw(self, stream: int, frames_ptr: int, n: int, scores_ptr=None, keep_ptr=None, hist_ptr=None,
                 cuda_stream=None):
        """The C entry point with plain addresses (device or host)."""
        st = self._stream(cuda_stream)
        rc = self._lib.cofie_ngff_push_ex(self._h, stream, frames_ptr, n, scores_ptr, keep_ptr, hist_ptr, st)
        self._check(rc)

    def make_batch(self, items):
        """Descriptor array for push_batch_raw from a list of
        (stream, frames[uint8], scores[f32] | None, keep[u8] | None), each
        tensor on the handle's device or in (preferably pinned) host memory."""
        arr = (_abi.PushDesc * max(1, len(items)))()
        for i, (stream, frames, scores, keep) in enumerate(items):
            n = self._frames(frames)
            arr[i].stream, arr[i].n = stream, n
            arr[i].frames, arr[i].scores_out, arr[i].keep_out = _ptr(frames), _ptr(scores), _ptr(keep)
        return arr, len(items)

    def push_batch(self, items, cuda_stream=None):
        """items: list of (stream, frames[uint8], scores[f32] | None, keep[u8] | None),
        device or host tensors; host frames of one call must fit one staging
        buffer (host_stage_bytes)."""
        arr, nd = self.make_batch(items)
        self.push_batch_raw(arr, nd, cuda_stream)

    def push_batch_raw(self, arr, nd: int, cuda_stream=None):
        """The batched C entry point on a prebuilt descriptor array."""
        self._check(self._lib.cofie_ngff_push_batch(self._h, arr, nd, self._stream(cuda_stream)))

    def candidates(self, stream: int = 0, cap: int | None = None, cuda_stream=None) -> torch.Tensor:
        """S_c of ``stream`` closed at the frames pushed so far, from the
        library's retention record: ascending indices (cuda int32) of the
        retained frames, the last frame and the M_min uniform fill.
        Synchronises to read the count. ``cap`` defaults to the frames seen."""
        if cap is None:
            cap = max(1, self.frames_seen(stream))
        idx = torch.empty(max(cap, 1), dtype=torch.int32, device=self.device)
        m = ctypes.c_uint32(0)
        self._check(self._lib.cofie_ngff_candidates(self._h, stream, _ptr(idx), cap, ctypes.addressof(m),
                                                    self._stream(cuda_stream)))
        if m.value > cap:
            raise ValueError(f"S_c has {m.value} frames, more than cap={cap}")
        return idx[: m.value]

    def candidates_raw(self, stream: int, idx_ptr: int, cap: int, m_ptr: int, cuda_stream=None):
        """The per-stream C entry point with plain device addresses (asynchronous)."""
        self._check(self._lib.cofie_ngff_candidates(self._h, stream, idx_ptr, cap, m_ptr, self._stream(cuda_stream)))

    def candidates_from_keep(self, keep: torch.Tensor, cuda_stream=None) -> torch.Tensor:
        """S_c of a prefix given by its keep codes (cuda uint8 in, cuda int32
        indices out; synchronises to read the count)."""
        T = keep.numel()
        idx = torch.empty(max(T, 1), dtype=torch.int32, device=self.device)
        m = ctypes.c_uint32(0)
        self._check(self._lib.cofie_ngff_candidates_from_keep(self._h, _ptr(keep), T, _ptr(idx), ctypes.addressof(m),
                                                              self._stream(cuda_stream)))
        return idx[: m.value]

    def gather(self, frames: torch.Tensor, idx: torch.Tensor, out: torch.Tensor | None = None, cuda_stream=None):
        """frames[idx] back to back (cuda uint8 [m, H, W, 3]): the encoder's input.
        frames may be on the device or in pinned host memory; idx is on the device."""
        n = self._frames(frames)
        m = idx.numel()
        if out is None:
            out = torch.empty((m, self.height, self.width, 3), dtype=torch.uint8, device=self.device)
        self._check(self._lib.cofie_ngff_gather(self._h, _ptr(frames), n, _ptr(idx), m, _ptr(out),
                                                self._stream(cuda_stream)))
        return out

    def state_save(self, stream: int = 0, out: torch.Tensor | None = None, cuda_stream=None) -> torch.Tensor:
        """The stream's saved state (uint8; host memory unless ``out`` is given)."""
        n = self._lib.cofie_ngff_state_bytes(self._h)
        if out is None:
            out = torch.empty(n, dtype=torch.uint8)
        self._check(self._lib.cofie_ngff_state_save(self._h, stream, _ptr(out), self._stream(cuda_stream)))
        return out

    def state_load(self, state: torch.Tensor, stream: int = 0, cuda_stream=None):
        self._check(self._lib.cofie_ngff_state_load(self._h, stream, _ptr(state), self._stream(cuda_stream)))

    def shard_prepare(self, frames_with_halo: torch.Tensor, n_halo: int, t0: int, stream: int = 0, cuda_stream=None):
        """Prepares one shard of a stream (halo frames then the shard's frames,
        cuda uint8); returns its gap map as a host int tensor of l_max entries."""
        n = self._frames(frames_with_halo) - n_halo
        m = torch.zeros(self.l_max, dtype=torch.int16)
        self._check(self._lib.cofie_ngff_shard_prepare(self._h, stream, _ptr(frames_with_halo), n_halo, n, t0,
                                                       _ptr(m), self._stream(cuda_stream)))
        return m.to(torch.int32)

    def shard_commit(self, entry_gap: int, n: int, stream: int = 0, cuda_stream=None):
        """Decides the prepared shard entered with ``entry_gap``; returns (scores, keep) on the device."""
        scores = torch.empty(n, dtype=torch.float32, device=self.device)
        keep = torch.empty(n, dtype=torch.uint8, device=self.device)
        self._check(self._lib.cofie_ngff_shard_commit(self._h, stream, entry_gap, _ptr(scores), _ptr(keep),
                                                      self._stream(cuda_stream)))
        return scores, keep

    def reset(self, stream: int = 0, cuda_stream=None):
        self._check(self._lib.cofie_ngff_reset(self._h, stream, self._stream(cuda_stream)))

    def status(self, cuda_stream=None):
        """Synchronises and raises NGFFError if a device-side wait ran out."""
        self._check(self._lib.cofie_ngff_status(self._h, self._stream(cuda_stream)))

    def frames_seen(self, stream: int = 0) -> int:
        t = ctypes.c_uint64(0)
        self._check(self._lib.cofie_ngff_frames_seen(self._h, stream, ctypes.byref(t)))
        return t.value

    def debug_bins(self, pixels: torch.Tensor, out: torch.Tensor | None = None, cuda_stream=None):
        """Device bin index of every RGB triple in ``pixels`` (cuda uint8 [..., 3])."""
        n = pixels.numel() // 3
        if out is None:
            out = torch.empty(n, dtype=torch.uint8, device=pixels.device)
        self._check(self._lib.cofie_ngff_debug_bins(self._h, _ptr(pixels), n, _ptr(out), self._stream(cuda_stream)))
        return out

    def debug_wait(self, timeout_ns: int, cuda_stream=None):
        """Enqueues the bounded-wait probe (a wait nothing completes); status()
        then raises NGFFError with code ETIMEOUT."""
        self._check(self._lib.cofie_ngff_debug_wait(self._h, int(timeout_ns), self._stream(cuda_stream)))

    def profile_reset(self, time_kernels: bool = False):
        """Zeroes the launch counters; with time_kernels every histogram-kernel
        launch is bracketed by CUDA events on its stream."""
        self._check(self._lib.cofie_ngff_profile_reset(self._h, int(time_kernels)))

    def profile_read(self) -> dict:
        pr = _abi.Profile()
        self._check(self._lib.cofie_ngff_profile_read(self._h, ctypes.byref(pr)))
        return {k: getattr(pr, k) for k, _ in _abi.Profile._fields_}

    def close(self):
        if getattr(self, "_h", None):
            self._lib.cofie_ngff_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 -- interpreter shutdown
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


class QER:
    """Query-specific evidence refinement (CoFiE Sec. 3.3) on the tensor cores:
    ranks candidate frames by text-to-vision attention and keeps the best
    max(1, round(rho m)) of them."""

    def __init__(self, n_text: int, n_heads: int, n_kv_heads: int, head_dim: int, max_frames: int,
                 tokens_per_frame: int, rho: float, device: int | None = None, kernel: int = 0):
        lib = _abi.load()
        p = _abi.QerParams(n_text, n_heads, n_kv_heads, head_dim, max_frames, tokens_per_frame, rho,
                           torch.cuda.current_device() if device is None else device, kernel)
        h = ctypes.c_void_p()
        rc = lib.cofie_qer_create(ctypes.byref(p), ctypes.byref(h))
        if rc != _abi.OK:
            raise NGFFError(rc, lib.cofie_qer_last_error(None).decode())
        self._lib, self._h, self.params = lib, h, p
        self.device = torch.device("cuda", p.device)
        self.kernel = int(lib.cofie_qer_kernel_in_use(h))  # 1: one-SM, 2: paired-SM

    def _check(self, rc):
        if rc != _abi.OK:
            raise NGFFError(rc, self._lib.cofie_qer_last_error(self._h).decode())

    def run(self, q: torch.Tensor, k: torch.Tensor, n_frames: int | None = None, cuda_stream=None):
        """q: bf16 bits (int16/uint16 or bfloat16) [n_text, H, d]; k: [n_frames * T, H_kv, d].
        Returns (w [n_frames] float32, selected frame indices int32, time order)."""
        T = self.params.tokens_per_frame
        n = k.shape[0] // T if n_frames is None else n_frames
        w = torch.empty(n, dtype=torch.float32, device=self.device)
        sel = torch.empty(n, dtype=torch.int32, device=self.device)
        kk = ctypes.c_uint32(0)
        st = torch.cuda.current_stream(self.device).cuda_stream if cuda_stream is None else int(cuda_stream)
        self._check(self._lib.cofie_qer_run(self._h, _ptr(q), _ptr(k), n, _ptr(w), _ptr(sel),
                                            ctypes.addressof(kk), st))
        return w, sel[: kk.value]

    def run_async(self, q: torch.Tensor, k: torch.Tensor, w: torch.Tensor, sel: torch.Tensor, k_dev: torch.Tensor,
                  n_frames: int | None = None, cuda_stream=None):
        """run() with every output in device memory (no synchronisation):
        w [n_frames] float32, sel [n_frames] int32 (first k_dev[0] entries valid)."""
        T = self.params.tokens_per_frame
        n = k.shape[0] // T if n_frames is None else n_frames
        st = torch.cuda.current_stream(self.device).cuda_stream if cuda_stream is None else int(cuda_stream)
        self._check(self._lib.cofie_qer_run(self._h, _ptr(q), _ptr(k), n, _ptr(w), _ptr(sel), _ptr(k_dev), st))

    def status(self, cuda_stream=None):
        st = torch.cuda.current_stream(self.device).cuda_stream if cuda_stream is None else int(cuda_stream)
        self._check(self._lib.cofie_qer_status(self._h, st))

    def profile_reset(self, time_kernels: bool = False):
        self._check(self._lib.cofie_qer_profile_reset(self._h, int(time_kernels)))

    def profile_read(self) -> dict:
        la, ti = ctypes.c_uint64(0), ctypes.c_uint64(0)
        ms, fl, kb = ctypes.c_double(0), ctypes.c_double(0), ctypes.c_double(0)
        self._check(self._lib.cofie_qer_profile_read(self._h, ctypes.byref(la), ctypes.byref(ti), ctypes.byref(ms),
                                                     ctypes.byref(fl), ctypes.byref(kb)))
        return {"launches": la.value, "timed": ti.value, "score_ms": ms.value, "flops": fl.value,
                "key_bytes": kb.value}

    def close(self):
        if getattr(self, "_h", None):
            self._lib.cofie_qer_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 -- interpreter shutdown
            pass
