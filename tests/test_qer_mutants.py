"""Plants one-spot mistakes in a copy of the QER oracle (on the CPU) and
checks that the pins of test_qer_oracle catch each of them."""
import pytest

from oracle import qer_oracle as Q
from tests import test_qer_oracle as PINS
from tests.mutation import call, caught_by, mutant, pins

MUTANTS = {
    "query head h reads key head h mod H_kv": ("a += (q[:, h, :] @ k[:, h // group, :].T) / np.sqrt(d)",
                                               "a += (q[:, h, :] @ k[:, h % H_kv, :].T) / np.sqrt(d)"),
    "scaled by 1/d": ("a += (q[:, h, :] @ k[:, h // group, :].T) / np.sqrt(d)",
                      "a += (q[:, h, :] @ k[:, h // group, :].T) / d"),
    "sum over heads, not mean": ("    return a / H\n", "    return a\n"),
    "mean over text tokens": ("best = a.max(axis=0)", "best = a.mean(axis=0)"),
    "max over the frame's tokens": ("best.reshape(-1, tokens_per_frame).mean(axis=1)",
                                    "best.reshape(-1, tokens_per_frame).max(axis=1)"),
    "frames strided over tokens": ("best.reshape(-1, tokens_per_frame).mean(axis=1)",
                                   "best.reshape(tokens_per_frame, -1).mean(axis=0)"),
    "k rounds half up": ("max(1, int(round(rho * n_frames)))", "max(1, int(rho * n_frames + 0.5))"),
    "k may be zero": ("max(1, int(round(rho * n_frames)))", "max(0, int(round(rho * n_frames)))"),
    "k truncated": ("max(1, int(round(rho * n_frames)))", "max(1, int(rho * n_frames))"),
    "ties to the later frame": ("key=lambda f: (-w[f], f)", "key=lambda f: (-w[f], -f)"),
    "lowest scores kept": ("key=lambda f: (-w[f], f)", "key=lambda f: (w[f], f)"),
    "rank order, not chronological": ("np.array(sorted(order[:k]), dtype=np.int64)",
                                      "np.array(order[:k], dtype=np.int64)"),
    "bound without the bf16 group rounding": ("rel = (2.0 ** -8 if group > 1 else 0.0)", "rel = (0.0)"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_each_mutant_is_caught(name, monkeypatch):
    monkeypatch.setattr(PINS, "Q", mutant(Q, *MUTANTS[name]))
    assert caught_by(PINS), f"mutant '{name}' passes every pin"


def test_unmutated_copy_passes_every_pin(monkeypatch):
    monkeypatch.setattr(PINS, "Q", mutant(Q, "    return a / H\n", "    return a / H\n"))
    for _, fn in pins(PINS):
        call(fn)
