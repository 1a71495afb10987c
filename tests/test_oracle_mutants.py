"""Plant one mistake at a time in a copy of the oracle and check that the
pins catch it: a dropped term, a wrong sign, a transposed operand, a wrong
bit index, a lost scale, a wrong spike test, a lost overflow check; for the
continuous-input projection a dropped row or activation stride, a dropped
term, a wrong sign, a lost scale, a signed magnitude, a float accumulator.  The
mutants are compiled on the CPU from the oracle's own source text."""
from pathlib import Path

import pytest

import oracle
from oracle_pins import ALL_PINS

SRC = (Path(oracle.__file__).parent / "spike_oracle.c").read_text()

MUTANTS = {
    "transposed_operand": ("Q[(int64_t)A[i] * ldq + m]", "Q[(int64_t)m * ldq + A[i]]"),
    "dropped_first_term": ("for (int32_t i = 0; i < nA; ++i)\n        acc +=",
                           "for (int32_t i = 1; i < nA; ++i)\n        acc +="),
    "wrong_sign": ("acc += Q[", "acc -= Q["),
    "bit_index_off_by_one": ("(k % 32)) & 1u", "((k + 1) % 32)) & 1u"),
    "msb_first_bits": ("(k % 32)) & 1u", "(31 - k % 32)) & 1u"),
    "scale_dropped": ("*y_out = s[m] * (float)acc32;", "*y_out = (float)acc32;"),
    "scale_of_wrong_channel": ("*y_out = s[m] * (float)acc32;", "*y_out = s[0] * (float)acc32;"),
    "u8_spike_is_exactly_one": ("((const uint8_t *)row)[k] != 0", "((const uint8_t *)row)[k] == 1"),
    "last_column_skipped": ("for (int32_t k = 0; k < K; ++k)\n        if (spike_at", "for (int32_t k = 0; k < K - 1; ++k)\n        if (spike_at"),
    "overflow_unchecked": ("if (acc > INT32_MAX || acc < INT32_MIN)\n        return -2;", ""),
    "narrow_accumulator": ("int64_t acc = 0;", "int16_t acc = 0;"),
    # continuous-input projection (every mutant stays inside its buffers)
    "dense_row_stride_ignored": ("const int8_t *q = Q + (int64_t)m * ldq;", "const int8_t *q = Q + (int64_t)m * K;"),
    "dense_x_stride_ignored": ("const float *xt = x + (int64_t)t * ldx;", "const float *xt = x + (int64_t)t * K;"),
    "dense_last_term_dropped": ("for (int32_t k = 0; k < K; ++k) {\n                double term", "for (int32_t k = 0; k + 1 < K; ++k) {\n                double term"),
    "dense_wrong_sign": ("dot += term;", "dot -= term;"),
    "dense_scale_dropped": ("y[(int64_t)t * N + m] = (double)s[m] * dot;", "y[(int64_t)t * N + m] = dot;"),
    "dense_abs_signed": ("mag += term < 0 ? -term : term;", "mag += term;"),
    "dense_float_accumulator": ("double dot = 0.0, mag = 0.0;", "float dot = 0.0f; double mag = 0.0;"),
    # spike producer (LIF step)
    "lif_multiply_then_add": ("float u = fmaf(beta, vt[k], it[k]);", "float u = beta * vt[k] + it[k];"),
    "lif_strict_threshold": ("if (u >= theta) {", "if (u > theta) {"),
    "lif_hard_reset": ("u = u - theta;", "u = 0.0f;"),
    "lif_no_reset": ("u = u - theta;", ""),
    "lif_msb_first": ("bt[k / 32] |= 1u << (k % 32);", "bt[k / 32] |= 1u << (31 - k % 32);"),
    "lif_tail_kept": ("for (int64_t w = 0; w < words; ++w)\n            bt[w] = 0u;", ""),
    "lif_row_stride_ignored": ("float *vt = v + (int64_t)t * ld;", "float *vt = v + (int64_t)t * K;"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    assert SRC.count(old) == 1, f"mutation site for {name} not unique"
    lib = oracle.compile_source(SRC.replace(old, new), tmp_path / "libmut.so")
    orc = oracle.Oracle(lib)
    failed = []
    for pin in ALL_PINS:
        try:
            pin(orc)
        except (AssertionError, RuntimeError):
            failed.append(pin.__name__)
    assert failed, f"no pin caught mutant {name}"
