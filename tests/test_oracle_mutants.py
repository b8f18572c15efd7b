"""Plants plausible mistakes in a copy of the oracle (on the CPU) and checks that the pin suite of
test_oracle_pins.py rejects every one of them: a dropped scale, a wrong group map, a block map
that picks the wrong layer, an off-by-one visible length, a missing normalisation, a flipped sign,
a wrong query row, a dropped factor in the cache size, a mis-numbered slot, a misplaced append,
a prefill row that does not see its own position, prefill queries read head-major, a merge that
drops the block's later layers, picks heads by a modulo group, sums without dividing, and a
bfloat16 rounding that truncates or rounds ties away from zero.
"""
import os
import subprocess
import tempfile

import pytest

import oracle
from oracle import build as oracle_build
import tests.test_oracle_pins as pins

MUTANTS = [
    ("no-scale", "work[t] = dot * inv_sqrt_dk;", "work[t] = dot;"),
    ("group-map-modulo", "int j = (i - 1) / (h / g) + 1;", "int j = (i - 1) % g + 1;"),
    ("block-owner-top", "int bottom = (k - 1) * per_block + 1;", "int bottom = k * per_block;"),
    ("visible-off-by-one", "int L = jb->seq_lens[beta];", "int L = jb->seq_lens[beta] - 1;"),
    ("no-normalisation", "work[t] = work[t] / Z;", "work[t] = work[t];"),
    ("flipped-exponent", "work[t] = exp(work[t] - smax);", "work[t] = exp(smax - work[t]);"),
    ("query-row-of-kv-head", "const double *q = jb->Q + ((size_t)beta * h + i) * d;",
     "const double *q = jb->Q + ((size_t)beta * h + j) * d;"),
    ("cache-size-drops-g", "return 2LL * b * s * m * g * dk;", "return 2LL * b * s * m * dk;"),
    ("slot-from-one", "slot[q] = m;", "slot[q] = m + 1;"),
    ("append-at-zero", "(size_t)(L - 1)) * d;", "(size_t)0) * d;"),
    ("prefill-excludes-self", "int L = t + 1;                     /* position t sees positions 0 .. t */",
     "int L = t > 0 ? t : 1;"),
    ("prefill-head-major-rows", "const double *q = jb->Q + (((size_t)beta * jb->s_max + t) * h + i) * d;",
     "const double *q = jb->Q + (((size_t)beta * h + i) * jb->s_max + t) * d;"),
    ("merge-owner-only", "                    if (owner[n] != o)\n                        continue;\n                    for (int i = j * G;",
     "                    if (n != o)\n                        continue;\n                    for (int i = j * G;"),
    ("merge-group-modulo", "for (int i = j * G; i < (j + 1) * G; ++i) {", "for (int i = j; i < h; i += g) {"),
    ("merge-sum-not-mean", "dst[r] = sum / (double)count;", "dst[r] = sum;"),
    ("bf16-truncates", "const double k = rint(ldexp(a, -q));", "const double k = trunc(ldexp(a, -q));"),
    ("bf16-ties-away", "const double k = rint(ldexp(a, -q));", "const double k = round(ldexp(a, -q));"),
]

PIN_TESTS = [
    pins.test_table2_total_kv_heads,
    pins.test_table1_opt175b_ratios_and_printed_values,
    pins.test_abstract_six_times_smaller_than_mqa,
    lambda: [pins.test_block_map_structure(l) for l in (2, 6, 12)],
    lambda: [pins.test_group_map(h) for h in (4, 12)],
    lambda: [pins.test_oracle_matches_sdpa(*m) for m in pins.MAPS],
    pins.test_mlkv_equals_mha_on_duplicated_kv,
    pins.test_single_position_returns_value_row,
    pins.test_equal_keys_and_zero_query_average_values,
    pins.test_dominant_key_selects_its_value,
    pins.test_brute_force_decimal,
    pins.test_append_only_for_owner_layers,
    lambda: [pins.test_prefill_matches_causal_sdpa(*m) for m in pins.MAPS],
    pins.test_prefill_first_position_returns_value_row,
    pins.test_merge_identity_map_returns_input,
    lambda: [pins.test_merge_linear_closed_form(*c) for c in
             [([0, 0, 0, 3, 3, 3], 12, 4), ([0, 0, 2, 2, 4, 4, 6, 6], 8, 1),
              ([0, 0, 0, 0, 4, 5, 5], 6, 3)]],
    pins.test_merge_permutation_invariance_and_locality,
    pins.test_bf16_rne_matches_torch_on_float32_values,
    pins.test_bf16_rne_brute_force_on_float64_values,
    pins.test_bf16_rne_worked_cases,
]


def _build_mutant(tmp, name, old, new):
    src = open(oracle_build.SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not unique"
    path_c = os.path.join(tmp, f"{name}.c")
    path_so = os.path.join(tmp, f"lib{name}.so")
    with open(path_c, "w") as f:
        f.write(src.replace(old, new))
    cmd = [c if c != oracle_build.SRC else path_c for c in oracle_build.command()]
    cmd = [c if c != oracle_build.LIB else path_so for c in cmd]
    subprocess.run(cmd, check=True)
    return path_so


def _pins_pass():
    for t in PIN_TESTS:
        try:
            t()
        except (AssertionError, ValueError):
            return False
    return True


def test_unmodified_oracle_passes_battery():
    assert _pins_pass()


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_reject_mutant(name, old, new):
    saved = oracle.lib()
    with tempfile.TemporaryDirectory() as tmp:
        try:
            oracle._lib = oracle.load(_build_mutant(tmp, name, old, new))
            assert not _pins_pass(), f"mutant {name} survived the pins"
        finally:
            oracle._lib = saved
