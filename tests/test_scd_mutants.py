"""Plants one-spot mistakes in a copy of the scene-change oracle (on the CPU)
and checks that the pins of test_scd_oracle catch each of them."""
import pytest

from oracle import scd_oracle as SC
from tests import test_scd_oracle as PINS
from tests.mutation import call, caught_by, mutant, pins

MUTANTS = {
    "cut does not end the run": ("            flags[t] = True\n            acc = 0\n",
                                 "            flags[t] = True\n"),
    "low difference does not end the run": ("        else:\n            acc = 0\n", "        else:\n            pass\n"),
    "fires on every frame past T_b": ("and not at_least(before, two_n, t_cut)", ""),
    "strict comparison": (">= np.float32(threshold)", "> np.float32(threshold)"),
    "scene change before novelty": (
        "        if at_least(max(na, nr), two_n, p.tau):\n            keep[t] = O.KEEP_NOVELTY\n"
        "        elif scene[t]:\n            keep[t] = KEEP_SCENE\n",
        "        if scene[t]:\n            keep[t] = KEEP_SCENE\n"
        "        elif at_least(max(na, nr), two_n, p.tau):\n            keep[t] = O.KEEP_NOVELTY\n"),
    "gap before scene change": (
        "        elif scene[t]:\n            keep[t] = KEEP_SCENE\n        elif p.l_max > 0 and t - r >= p.l_max:\n"
        "            keep[t] = O.KEEP_GAP\n",
        "        elif p.l_max > 0 and t - r >= p.l_max:\n            keep[t] = O.KEEP_GAP\n        elif scene[t]:\n"
        "            keep[t] = KEEP_SCENE\n"),
    "scene keeps do not move r": ("        if keep[t]:\n            r = t\n",
                                  "        if keep[t] and keep[t] != KEEP_SCENE:\n            r = t\n"),
    "gradual threshold used for the cut": ("    if at_least(a, two_n, t_cut):\n        return HIGH",
                                           "    if at_least(a, two_n, t_grad):\n        return HIGH"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_each_mutant_is_caught(name, monkeypatch):
    monkeypatch.setattr(PINS, "SC", mutant(SC, *MUTANTS[name]))
    assert caught_by(PINS), f"mutant '{name}' passes every pin"


def test_unmutated_copy_passes_every_pin(monkeypatch):
    monkeypatch.setattr(PINS, "SC", mutant(SC, "KEEP_SCENE = 4", "KEEP_SCENE = 4"))
    for _, fn in pins(PINS):
        call(fn)
