"""Plausible mistakes planted in a copy of the oracle must each fail a pin.

Every mutant below is a one-spot edit of ngff_oracle.c (a dropped term, a
wrong operand, index or comparison). The copy is compiled into a temporary
directory and the whole pin suite runs against it in a child process; the
test passes only if at least one pin fails. The real oracle is untouched.
"""
import os
import subprocess
import sys

import pytest

import oracle
from tests.conftest import REPO

SRC = os.path.join(REPO, "oracle", "ngff_oracle.c")

MUTANTS = {
    "luma_r_b_swapped": ("(uint64_t)p->luma_w[0] * r + (uint64_t)p->luma_w[1] * g + (uint64_t)p->luma_w[2] * b",
                         "(uint64_t)p->luma_w[0] * b + (uint64_t)p->luma_w[1] * g + (uint64_t)p->luma_w[2] * r"),
    "luma_no_rounding": ("(num + p->luma_den / 2) / p->luma_den", "num / p->luma_den"),
    "luma_round_down_at_half": ("(num + p->luma_den / 2) / p->luma_den", "(num + p->luma_den / 2 - 1) / p->luma_den"),
    "bin_divisor_257": ("(y * bins) / 256u", "(y * bins) / 257u"),
    "hist_reads_bgr": ("ngff_oracle_luma(px[0], px[1], px[2], p)", "ngff_oracle_luma(px[2], px[1], px[0], p)"),
    "tv_no_half": ("return 0.5 * acc;", "return acc;"),
    "tv_signed_sum": ("acc += hi > hj ? hi - hj : hj - hi;", "acc += hi - hj;"),
    "tv32_over_n": ("volatile float den = (float)(2 * npix);", "volatile float den = (float)(npix);"),
    "adj_compares_self": ("double s_adj = ngff_oracle_tv(ht, hist + (size_t)(t - 1) * B, B, N);",
                          "double s_adj = ngff_oracle_tv(ht, hist + (size_t)(t) * B, B, N);"),
    "adj32_compares_self": ("float d_adj = ngff_oracle_tv32(ht, hist + (size_t)(t - 1) * B, B, N);",
                            "float d_adj = ngff_oracle_tv32(ht, hist + (size_t)(t) * B, B, N);"),
    "ref_is_first_frame": ("float d_ref = ngff_oracle_tv32(ht, hist + (size_t)r * B, B, N);",
                           "float d_ref = ngff_oracle_tv32(ht, hist, B, N);"),
    "min_not_max": ("float s32 = d_adj > d_ref ? d_adj : d_ref;", "float s32 = d_adj < d_ref ? d_adj : d_ref;"),
    "score_min_not_max": ("score = s_adj > s_ref ? s_adj : s_ref;", "score = s_adj < s_ref ? s_adj : s_ref;"),
    "strict_tau": ("int novelty = s32 >= p->tau;", "int novelty = s32 > p->tau;"),
    "strict_gap": ("int gap = p->l_max > 0 && (t - r) >= p->l_max;", "int gap = p->l_max > 0 && (t - r) > p->l_max;"),
    "gap_off_by_one": ("int gap = p->l_max > 0 && (t - r) >= p->l_max;",
                       "int gap = p->l_max > 0 && (t - r) >= p->l_max + 1;"),
    "gap_rule_with_zero_l_max": ("int gap = p->l_max > 0 && (t - r) >= p->l_max;", "int gap = (t - r) >= p->l_max;"),
    "r_not_moved_by_gap": ("if (keep != KEEP_DROP) r = t;", "if (keep == KEEP_NOVELTY || keep == KEEP_FIRST) r = t;"),
    "first_not_kept": ("keep = KEEP_FIRST; /* the first", "keep = KEEP_DROP; /* the first"),
    "gap_code_wins": ("keep = novelty ? KEEP_NOVELTY : (gap ? KEEP_GAP : KEEP_DROP);",
                      "keep = gap ? KEEP_GAP : (novelty ? KEEP_NOVELTY : KEEP_DROP);"),
    "last_not_added": ("in[T - 1] = 1; /* the last", "/* the last"),
    "fill_floor": ("uint64_t num = 2ull * i * (T - 1) + (m_min - 1);", "uint64_t num = 2ull * i * (T - 1);"),
    "fill_when_equal": ("if (count < m_min) {", "if (count <= m_min) {"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    msrc = tmp_path / "mutant.c"
    msrc.write_text(src.replace(old, new))
    lib = str(tmp_path / "libmutant.so")
    oracle.build(force=True, src=str(msrc), out=lib)
    r = subprocess.run([sys.executable, os.path.join(REPO, "tests", "oracle_pins.py"), lib],
                       capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"no pin caught mutant {name}:\n{r.stdout}\n{r.stderr}"
