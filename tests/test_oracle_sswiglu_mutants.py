"""Mutation check of the Spatial SwiGLU oracle's pins (Eq. spatial_swiglu): plausible
mistakes are planted in a copy of oracle.sswiglu_dwconv (on the CPU), and at least
one of its pins in tests/test_oracle_pins.py must fail against the copy."""
import inspect
import textwrap

import numpy as np
import pytest

import oracle
import test_oracle_pins as pins

MUTANTS = {
    # a convolution with the kernel flipped instead of the layer's cross-correlation
    "kernel_flipped": ("conv += w[:, i, j] * pad[", "conv += w[:, 2 - i, 2 - j] * pad["),
    # row and column offsets of the taps swapped
    "taps_transposed": ("conv += w[:, i, j] * pad[", "conv += w[:, j, i] * pad["),
    # tokens read in column-major order
    "grid_transposed": ("img = v.reshape(B, grid_h, grid_w, F)",
                        "img = v.reshape(B, grid_w, grid_h, F).transpose(0, 2, 1, 3)"),
    # the bias dropped
    "no_bias": ("conv += np.asarray(bias, dtype=np.float64)", "pass"),
    # SiLU with the sign of the exponent flipped
    "silu_sign": ("silu = g / (1.0 + np.exp(-g))", "silu = g / (1.0 + np.exp(g))"),
    # periodic instead of zero padding
    "wrap_padding": ("pad[:, 1:grid_h + 1, 1:grid_w + 1, :] = img",
                     "pad = np.pad(img, ((0, 0), (1, 1), (1, 1), (0, 0)), mode='wrap')"),
    # column taps shifted by one
    "column_offset": ("pad[:, i:i + grid_h, j:j + grid_w, :]",
                      "pad[:, i:i + grid_h, (j + 1) % 3:(j + 1) % 3 + grid_w, :]"),
    # the bias added after the gate instead of to the convolution
    "bias_after_gate": ("return silu * conv.reshape(B, T, F)",
                        "return silu * (conv.reshape(B, T, F) - (0 if bias is None else np.asarray(bias))) + "
                        "(0 if bias is None else np.asarray(bias))"),
}

PINS = [pins.test_sswiglu_hand_worked_2x3, pins.test_sswiglu_matches_scipy_correlate2d,
        pins.test_sswiglu_special_cases]


def _mutant(old, new):
    src = textwrap.dedent(inspect.getsource(oracle.sswiglu_dwconv))
    assert src.count(old) == 1, old
    ns = {}
    exec(compile(src.replace(old, new), "<mutant>", "exec"), vars(oracle).copy(), ns)
    return ns["sswiglu_dwconv"]


def test_pins_pass_on_the_oracle():
    pytest.importorskip("scipy.signal")
    for pin in PINS:
        pin()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_some_pin_catches_mutant(name, monkeypatch):
    pytest.importorskip("scipy.signal")
    monkeypatch.setattr(oracle, "sswiglu_dwconv", _mutant(*MUTANTS[name]))
    failed = []
    for pin in PINS:
        try:
            pin()
        except AssertionError:
            failed.append(pin.__name__)
    assert failed, f"mutant {name} passed every pin"
