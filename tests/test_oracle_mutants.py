"""Plant one mistake at a time in a copy of the oracle and check that the
pins catch it: a dropped term, a wrong sign, a transposed operand, a wrong
bit index, a lost scale, a wrong spike test, a lost overflow check; for the
continuous-input projection a dropped row or activation stride, a dropped
term, a wrong sign, a lost scale, a signed magnitude, a float accumulator;
for the LIF step and the vocabulary head the mistakes listed by name.  The
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
    # vocabulary head (every mutant stays inside its buffers; the comparator
    # mutants stay consistent orders)
    "head_scale_without_127": ("fmaxf(amax, 1e-8f) / 127.0f", "fmaxf(amax, 1e-8f) / 128.0f"),
    "head_no_floor": ("const float sx = fmaxf(amax, 1e-8f)", "const float sx = fmaxf(amax, 1e-12f)"),
    "head_truncating_round": ("float c = rintf(hb[k] / sx);", "float c = truncf(hb[k] / sx);"),
    "head_round_half_away": ("float c = rintf(hb[k] / sx);", "float c = roundf(hb[k] / sx);"),
    "head_clip_126": ("if (c > 127.0f)\n                c = 127.0f;", "if (c > 126.0f)\n                c = 126.0f;"),
    "head_last_column_dropped": ("for (int32_t k = 0; k < K; ++k)\n                a += ", "for (int32_t k = 0; k + 1 < K; ++k)\n                a += "),
    "head_row_stride_ignored": ("const int8_t *row = Q + (int64_t)m * ldq;\n            int64_t a = 0;", "const int8_t *row = Q + (int64_t)m * K;\n            int64_t a = 0;"),
    "head_h_stride_ignored": ("const float *hb = h + (int64_t)b * ldh;", "const float *hb = h + (int64_t)b * K;"),
    "head_scale_of_wrong_row": ("order[m].z = s[m] * t;", "order[m].z = s[0] * t;"),
    "head_ascending_order": ("if (a->z > b->z)\n        return -1;\n    if (a->z < b->z)\n        return 1;", "if (a->z < b->z)\n        return -1;\n    if (a->z > b->z)\n        return 1;"),
    "head_ties_by_higher_index": ("return a->m < b->m ? -1 : (a->m > b->m ? 1 : 0);", "return a->m > b->m ? -1 : (a->m < b->m ? 1 : 0);"),
    "head_gap_to_third": ("const float g = order[0].z - order[1].z;", "const float g = order[0].z - order[2].z;"),
    "head_gate_inclusive": ("const int open = g < tau;", "const int open = g <= tau;"),
    "head_verify_from_codes": ("const double term = (double)row[k] * (double)hb[k];", "const double term = (double)row[k] * (double)q[k] * (double)sx;"),
    "head_verify_scale_dropped": ("rc[i] = (double)s[m] * sum;", "rc[i] = sum;"),
    "head_token_never_verified": ("token[b] = open ? order[best].m : order[0].m;", "token[b] = order[0].m;"),
    "head_token_tie_higher": ("(rc[i] == rc[best] && m < order[best].m)", "(rc[i] == rc[best] && m > order[best].m)"),
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
