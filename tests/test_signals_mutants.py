"""Plants one-spot mistakes in a copy of the alternative-signal oracle (on the
CPU) and checks that the pins of test_signals_oracle catch each of them."""
import pytest

from oracle import signals_oracle as SO
from tests import test_signals_oracle as PINS
from tests.mutation import call, caught_by, mutant, pins

BITS = "bits = S[:, :-1] * n[:, 1:] > S[:, 1:] * n[:, :-1]"

MUTANTS = {
    "dHash bit on equal means": (BITS, "bits = S[:, :-1] * n[:, 1:] >= S[:, 1:] * n[:, :-1]"),
    "dHash compares sums, not means": (BITS, "bits = S[:, :-1] > S[:, 1:]"),
    "dHash compares down the columns": (BITS, "bits = S[:-1, :] * n[1:, :] > S[1:, :] * n[:-1, :]"),
    "dHash grid transposed": ("DHASH: (8, 9)", "DHASH: (9, 8)"),
    "cell index rounded up": ("cy = (np.arange(H) * gh) // H", "cy = (np.arange(H) * gh + H - 1) // H"),
    "low-res denominator 2N": ("255 * p.npix if kind == LOWRES", "2 * p.npix if kind == LOWRES"),
    "low-res signed difference": ("int(np.abs(fa - fb).sum())", "int((fa - fb).sum())"),
    "Hamming counts equal bits": ("int((fa != fb).sum())", "int((fa == fb).sum())"),
    "adjacent term dropped": ("na = numerator(feats[t], feats[t - 1], kind)", "na = 0"),
    "reference term dropped": ("nr = numerator(feats[t], feats[r], kind)", "nr = 0"),
    "reference never moves": ("        if keep[t]:\n            r = t\n", "        if keep[t]:\n            pass\n"),
    "strict novelty comparison": ("nov = s32 >= np.float32(p.tau)", "nov = s32 > np.float32(p.tau)"),
    "gap one frame late": ("(t - r) >= p.l_max", "(t - r) > p.l_max"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_each_mutant_is_caught(name, monkeypatch):
    monkeypatch.setattr(PINS, "SO", mutant(SO, *MUTANTS[name]))
    assert caught_by(PINS), f"mutant '{name}' passes every pin"


def test_unmutated_copy_passes_every_pin(monkeypatch):
    monkeypatch.setattr(PINS, "SO", mutant(SO, "LOWRES, DHASH = 1, 2", "LOWRES, DHASH = 1, 2"))
    for _, fn in pins(PINS):
        call(fn)
