"""ORACLE for query-specific evidence refinement (QER), CoFiE Sec. 3.3 --
test infrastructure only.

A plain numpy (float64) restatement of Eqs. 6-8, in the paper's order. Only
the tests and the benchmark's CPU-baseline leg use it; the GPU library shares
no code with it. A matrix product (numpy matmul) serves as a library step.

  Eq. 6  a_ij = (1/H) sum_h <q_i^h, k_j^h> / sqrt(d_h)   for text token i and
         visual token j. Reading for grouped key/value heads (the backbone's
         attention has H query heads and H_kv < H key heads): query head h
         reads key head h // (H / H_kv), as in the attention itself.
  Eq. 7  w_f = (1 / |V_f|) sum_{j in V_f} max_{i in Q} a_ij, V_f the frame's
         tokens (a contiguous run of tokens_per_frame keys per frame).
  Eq. 8  k = max(1, round(rho |S_c|)), S_e = TopK_f (w_f, k), returned in
         chronological order. Readings: round() rounds half to even (Python's
         round and torch.round); equal scores are ranked by lower frame index.

Inputs are bf16 bit patterns (uint16), converted exactly.
"""
from __future__ import annotations

import numpy as np


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def token_scores(q_bits: np.ndarray, k_bits: np.ndarray) -> np.ndarray:
    """Eq. 6: a [n_text, n_visual] from q [n_text, H, d] and k [n_visual, H_kv, d]."""
    q = bf16_to_f64(q_bits)
    k = bf16_to_f64(k_bits)
    n_text, H, d = q.shape
    H_kv = k.shape[1]
    assert H % H_kv == 0 and k.shape[2] == d
    group = H // H_kv
    a = np.zeros((n_text, k.shape[0]), dtype=np.float64)
    for h in range(H):
        a += (q[:, h, :] @ k[:, h // group, :].T) / np.sqrt(d)
    return a / H


def frame_relevance(a: np.ndarray, tokens_per_frame: int) -> np.ndarray:
    """Eq. 7: max over text tokens, then mean over each frame's tokens."""
    best = a.max(axis=0)
    return best.reshape(-1, tokens_per_frame).mean(axis=1)


def keep_count(n_frames: int, rho: float) -> int:
    """Eq. 8: k = max(1, round(rho * |S_c|)), round half to even."""
    return max(1, int(round(rho * n_frames)))


def select(w: np.ndarray, rho: float) -> np.ndarray:
    """Eq. 8: the k best frames by w (ties: lower index first), chronological."""
    k = keep_count(len(w), rho)
    order = sorted(range(len(w)), key=lambda f: (-w[f], f))
    return np.array(sorted(order[:k]), dtype=np.int64)


def run(q_bits, k_bits, tokens_per_frame: int, rho: float):
    """Eqs. 6-8 end to end: (w [n_frames], S_e)."""
    w = frame_relevance(token_scores(q_bits, k_bits), tokens_per_frame)
    return w, select(w, rho)


def frame_relevance_subset(q_bits, k_bits, tokens_per_frame: int, frames) -> np.ndarray:
    """Eq. 7 for the listed frames only (Eq. 6 restricted to their tokens)."""
    out = []
    for f in frames:
        sl = slice(int(f) * tokens_per_frame, (int(f) + 1) * tokens_per_frame)
        out.append(frame_relevance(token_scores(q_bits, k_bits[sl]), tokens_per_frame)[0])
    return np.array(out)


def score_bound(q_bits, k_bits, tokens_per_frame: int, frames=None) -> np.ndarray:
    """An upper bound on |w_f(computed) - w_f| for a computation that sums the
    query heads of each key/value group, rounds that sum to bf16 (relative
    error <= 2^-8, only when a group has more than one head), and accumulates
    the D = H_kv * d products in fp32 (relative error <= D * 2^-23): per token
    pair rel * (1/(H sqrt(d))) sum_{h,k} |q_i^h[k]| |k_j^{h}[k]|; the max over
    text and the mean over the frame's tokens keep the bound."""
    q = np.abs(bf16_to_f64(q_bits))
    k = np.abs(bf16_to_f64(k_bits))
    n_text, H, d = q.shape
    group = H // k.shape[1]
    rel = (2.0 ** -8 if group > 1 else 0.0) + k.shape[1] * d * 2.0 ** -23
    frames = range(k.shape[0] // tokens_per_frame) if frames is None else frames
    out = []
    for f in frames:
        sl = slice(int(f) * tokens_per_frame, (int(f) + 1) * tokens_per_frame)
        b = np.zeros((n_text, tokens_per_frame))
        for h in range(H):
            b += q[:, h, :] @ k[sl, h // group, :].T
        out.append(rel * (b / (H * np.sqrt(d))).max(axis=0).mean())
    return np.array(out)
