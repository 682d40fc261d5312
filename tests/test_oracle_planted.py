"""Planted mistakes: each mutant is the oracle's C source with one plausible
error written in; compiled on the CPU into a temporary library, it must fail
at least one pin.  This shows the pins can tell a wrong oracle from the real
one (the real one passes them all in test_oracle_pins.py)."""
import os
import subprocess

import pytest

import oracle
import pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "vd_oracle.c")

MUTANTS = {
    # the mean over n-1 tokens instead of n (Eq. vd)
    "mean_divisor": ("out[c] /= (double)n;", "out[c] /= (double)(n - 1);"),
    # the mean leaves out the newest token
    "mean_drops_last_row": ("for (int64_t i = 0; i < n; ++i) {\n      double x = vdo_bf16_to_double(v[i * d + c]);",
                            "for (int64_t i = 0; i < n - 1; ++i) {\n      double x = vdo_bf16_to_double(v[i * d + c]);"),
    # v_j + mean instead of v_j - mean
    "l2_sign": ("double diff = vdo_bf16_to_double(row[c]) - mean[c];",
                "double diff = vdo_bf16_to_double(row[c]) + mean[c];"),
    # squared distance reported as the score
    "l2_no_sqrt": ("out[j] = sqrt(acc);", "out[j] = acc;"),
    # Dir normalised by the wrong norm
    "dir_wrong_norm": ("dot / (vnorm * mean_norm)", "dot / (vnorm * vnorm)"),
    # Dir reports cos instead of 1 - cos
    "dir_cos": ("out[j] = 1.0 - cosv;", "out[j] = cosv;"),
    # Norm reports the squared norm
    "norm_squared": ("out[j] = sqrt(vv);", "out[j] = vv;"),
    # keeps the lowest scores
    "keeps_lowest": ("if (a->score > b->score) return -1;", "if (a->score < b->score) return -1;"),
    # ties go to the higher index
    "tie_to_higher_index": ("return (a->index > b->index) - (a->index < b->index);",
                            "return (a->index < b->index) - (a->index > b->index);"),
    # kept list left in score order instead of slot order
    "kept_not_ascending": ("qsort(kept, (size_t)N, sizeof(int32_t), vdo_int_cmp);", "(void)vdo_int_cmp;"),
    # V gathered from K's rows (transposed operand)
    "gather_wrong_tensor": ("memcpy(vv + r * d, v + (int64_t)idx[r] * d, row_bytes);",
                            "memcpy(vv + r * d, k + (int64_t)idx[r] * d, row_bytes);"),
    # FastCAOTE factor a/(1+a) instead of a/(1-a)
    "weight_factor": ("out[j] *= a[j] / (1.0 - a[j]);", "out[j] *= a[j] / (1.0 + a[j]);"),
    # sample standard deviation instead of the population one
    "dispersion_divisor": ("return sqrt(ss / (double)n);", "return sqrt(ss / (double)(n - 1));"),
    # gather off by one row
    "gather_off_by_one": ("memcpy(kk + r * d, k + (int64_t)idx[r] * d, row_bytes);",
                          "memcpy(kk + r * d, k + (int64_t)(idx[r] > 0 ? idx[r] - 1 : 0) * d, row_bytes);"),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(tmp_path, source, name):
    find, repl = MUTANTS[name]
    assert source.count(find) == 1, f"mutation site for {name} not unique in the oracle source"
    mutated = tmp_path / "vd_oracle.c"
    mutated.write_text(source.replace(find, repl))
    lib = tmp_path / "libmutant.so"
    oracle.build(force=True, src=str(mutated), out=str(lib))
    failures = pins.all_checks(oracle.load(str(lib)))
    assert failures, f"planted mistake {name!r} passed every pin"


def test_real_oracle_passes_every_pin(orc):
    assert pins.all_checks(orc) == []
