"""Mutation check of the oracle's pins: plausible mistakes are planted in a
copy of oracle/gla_oracle.c (on the CPU), the copy is compiled, and at least
one pin of tests/test_oracle_pins.py must fail against it."""
import os
import shutil
import subprocess

import pytest

import oracle
import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "gla_oracle.c")

MUTANTS = {
    # decay also applied to the incoming token's k^T v
    "decay_after_add": ("S[i * Dv + j] = gamma * S[i * Dv + j] + kt[i] * vt[j];",
                        "S[i * Dv + j] = gamma * (S[i * Dv + j] + kt[i] * vt[j]);"),
    # column scan with the grid sides swapped
    "col_scan_transposed": ("case ORDER_COL_FWD: return (s % grid_h) * grid_w + s / grid_h;",
                            "case ORDER_COL_FWD: return (s % grid_w) * grid_h + s / grid_w;"),
    # reverse column scan walking each column bottom-up from column 0
    "col_rev_per_column": ("return (u % grid_h) * grid_w + u / grid_h;",
                           "return (grid_h - 1 - s % grid_h) * grid_w + s / grid_h;"),
    # gate read from the value side
    "gate_on_value_side": ("double gamma = exp(gt[i]);",
                           "double gamma = exp(gt[i < Dv ? i : 0]) * 0 + exp(gt[0]);"),
    # chunk output: strict mask (drops the j = r term)
    "chunk_strict_mask": ("for (long j = 0; j <= r; ++j) {", "for (long j = 0; j < r; ++j) {"),
    # chunk readout with the exclusive cumulative decay
    "chunk_exclusive_readout": ("acc += qr[i] * exp(A[r * Dk + i]) * S[i * Dv + jv];",
                                "acc += qr[i] * exp(r > 0 ? A[(r - 1) * Dk + i] : 0.0) * S[i * Dv + jv];"),
    # chunk summary decays from the wrong end
    "chunk_summary_flipped": ("double khat = kr[i] * exp(A[(Cc - 1) * Dk + i] - A[r * Dk + i]);",
                              "double khat = kr[i] * exp(A[r * Dk + i]);"),
    # boundary state not decayed
    "chunk_no_state_decay": ("S[i * Dv + jv] = d * S[i * Dv + jv] + U[i * Dv + jv];",
                             "S[i * Dv + jv] = S[i * Dv + jv] + U[i * Dv + jv];"),
    # readout with S transposed (only differs when Dk != Dv)
    "readout_transposed": ("for (long i = 0; i < Dk; ++i) acc += qt[i] * S[i * Dv + j];",
                           "for (long i = 0; i < Dk && i < Dv && j < Dk; ++i) acc += qt[i] * S[j * Dv + i];"),
}

PIN_CHECKS = [
    lambda: pins.test_scan_orders_match_hand_lists(),
    lambda: pins.test_hand_worked_recurrence("row_fwd", oracle.ROW_FWD),
    lambda: pins.test_hand_worked_recurrence("row_rev", oracle.ROW_REV),
    lambda: pins.test_hand_worked_chunkwise("row_fwd", oracle.ROW_FWD, 2),
    lambda: [pins.test_brute_force_quadratic_form(o, 3, 5) for o in range(4)],
    lambda: [pins.test_brute_force_quadratic_form(o, 4, 2) for o in range(4)],
    lambda: pins.test_chunk_size_invariance(7, 3),
]


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(name, tmp_path):
    before, after = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(before) == 1, f"mutation site for {name} not found exactly once"
    mutant = tmp_path / "mutant.c"
    mutant.write_text(src.replace(before, after))
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fopenmp", "-shared", "-fPIC", "-o", str(so),
                    str(mutant), "-lm"], check=True)
    failures = 0
    with oracle.using_library(str(so)):
        for check in PIN_CHECKS:
            try:
                check()
            except AssertionError:
                failures += 1
    assert failures > 0, f"no pin caught mutant {name}"
