"""Seeded synthetic inputs for query-specific evidence refinement (QER).

Input generation only: this module holds none of the method's arithmetic. It
draws bf16 text queries Q [n_text, H, d] and visual keys K [n_frames *
tokens_per_frame, H_kv, d] (as uint16 bit patterns, round-to-nearest-even
from float32 draws) shaped like the last-layer attention inputs of
Qwen3-VL-8B (H = 32 query heads, H_kv = 8 key/value heads, d = 128), which
stand in for the model the paper uses. A few "evidence" frames get a key
component aligned with one text query, so that the frame ranking has a
planted answer.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class QerSpec:
    n_text: int = 256
    n_heads: int = 32
    n_kv_heads: int = 8
    head_dim: int = 128
    n_frames: int = 128
    tokens_per_frame: int = 256
    n_evidence: int = 8
    seed: int = 0xC0F1E0A0
    integer: bool = False  # small integers in [-4, 4]: every product and sum is exact in fp32

    @property
    def n_visual(self) -> int:
        return self.n_frames * self.tokens_per_frame

    def with_(self, **kw) -> "QerSpec":
        d = self.__dict__.copy()
        d.update(kw)
        return QerSpec(**d)


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return b.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float32, exactly."""
    return (b.astype(np.uint32) << 16).view(np.float32)


def generate(spec: QerSpec):
    """Returns (q_bits [n_text, H, d] uint16, k_bits [n_visual, H_kv, d] uint16,
    evidence_frames sorted int array)."""
    g = np.random.Generator(np.random.Philox(spec.seed))
    if spec.integer:
        q = g.integers(-4, 5, size=(spec.n_text, spec.n_heads, spec.head_dim)).astype(np.float32)
        k = g.integers(-4, 5, size=(spec.n_visual, spec.n_kv_heads, spec.head_dim)).astype(np.float32)
        return to_bf16_bits(q), to_bf16_bits(k), np.zeros(0, dtype=np.int64)
    q = g.standard_normal((spec.n_text, spec.n_heads, spec.head_dim), dtype=np.float32)
    k = g.standard_normal((spec.n_visual, spec.n_kv_heads, spec.head_dim), dtype=np.float32)
    ev = np.sort(g.choice(spec.n_frames, size=min(spec.n_evidence, spec.n_frames), replace=False))
    group = spec.n_heads // spec.n_kv_heads
    for f in ev:
        i = int(g.integers(spec.n_text))
        # keys of the frame's tokens lean towards text token i (its heads averaged per key/value group)
        target = q[i].reshape(spec.n_kv_heads, group, spec.head_dim).mean(axis=1)
        target /= np.linalg.norm(target, axis=-1, keepdims=True)
        sl = slice(f * spec.tokens_per_frame, (f + 1) * spec.tokens_per_frame)
        k[sl] += 1.5 * target[None, :, :] * np.sqrt(spec.head_dim) / 4
    return to_bf16_bits(q), to_bf16_bits(k), ev
