"""Pins for the CPU oracle: checks against facts fixed by the paper and by
arithmetic, not by the oracle itself.

Each ``pin_*`` takes an ``oracle.Oracle`` and raises ``AssertionError`` when
the oracle disagrees.  ``test_oracle_pins.py`` runs them on the real oracle;
``test_oracle_mutants.py`` runs them on copies of the oracle with one planted
mistake each and requires every copy to fail at least one pin.

What pins what (Section 2.3, Eq. sparse: y_m = s_m * sum_{k in A} Q_{m,k}):

* hand-worked fixture (tests/golden/hand_worked.json) -- values worked out by
  hand from the equation;
* exhaustive masks and full shapes -- the sum over A equals the dense
  integer product Q x for binary x (numpy int64 matmul, a library routine);
* the scale -- one FP32 multiply of an exactly converted integer is the
  correctly rounded exact product (fp64 holds acc*s exactly: 24 + 24 bits);
* invariants -- zero spikes, one-hot, additivity over disjoint sets,
  all-ones row sums, column permutation, format equivalence, tail bits,
  nonzero bytes;
* closed forms -- constant Q, INT8 extremes, INT32 overflow reported.

The continuous-input projection (Section 2.3, row-major weights of Section
2.2: y_m = s_m * sum_k Q[m][k] x_k, evaluated in double) is pinned by a
hand-worked fixture (tests/golden/hand_worked_dense.json), numpy float64
matmul with padded row strides, closed forms (constant Q and x, one-hot,
zero, extremes), linearity on dyadic inputs (exact in double), and, for
0/1 inputs, exact agreement with the spike-gated projection of the same
matrix.

The spike producer (one LIF step of the stated reading, written as BITS32
rows) is pinned by a hand-worked fixture (tests/golden/hand_worked_lif.json),
an exactly periodic closed form, cases where a fused multiply-add and a
separate multiply then add round differently (exact rational arithmetic
rounded to FP32), the bit format and cleared tail bits via the spike
oracle's own unpacking, row strides, and an infinite threshold.

The vocabulary head (INT8 activations, top-two gap gate, FP32-activation
recompute of the top candidates) is pinned by a hand-worked fixture
(tests/golden/hand_worked_head.json) in which verification changes the
token and an exact tie picks the lower index; activations that are exact
INT8 codes times a power of two (the recompute must then equal the
approximate logit and the numpy integer product); round-half-even codes and
the 1e-8 floor; numpy's lexsort of the logits with duplicate rows and the
strict gate at tau = gap; row and column permutations; the dense oracle's
projection and argmax when every row is a candidate; and the zero state.
"""
from __future__ import annotations

import json
from pathlib import Path

import numpy as np

from paper_2606_03026_gb300 import synth

GOLDEN = Path(__file__).resolve().parent / "golden"


def logical(Qc: np.ndarray, N: int) -> np.ndarray:
    """Logical [N, K] view of column-major storage [K, ldq]."""
    return np.asarray(Qc)[:, :N].T.astype(np.int64)


def dense_ref(Qc, N, x_u8):
    """Dense integer product Q x for each binary row of x (numpy int64)."""
    return (np.asarray(x_u8, dtype=np.int64) != 0).astype(np.int64) @ logical(Qc, N).T


def f32_bits(a):
    return np.asarray(a, dtype=np.float32).view(np.uint32)


def exact_scaled(acc, s):
    """Correctly rounded fp32 of the exact product acc * s (fp64 is exact
    here: |acc| < 2^24 and s has a 24-bit significand)."""
    return (np.asarray(acc, np.float64) * np.asarray(s, np.float32).astype(np.float64)).astype(np.float32)


# --------------------------------------------------------------------------
def pin_hand_fixture(orc):
    g = json.loads((GOLDEN / "hand_worked.json").read_text())
    N, K, ldq = g["N"], g["K"], g["ldq"]
    rows = np.array(g["Q_logical_rows_m_by_k"], dtype=np.int64)
    Qc = np.full((K, ldq), g["pad_byte"], dtype=np.int8)
    Qc[:, :N] = rows.T.astype(np.int8)
    s = np.array(g["scale"], dtype=np.float32)
    for case in g["cases"]:
        want_acc = np.array(case["acc"], dtype=np.int32)
        want_y = np.array(case["y"], dtype=np.float32)
        x = np.array(case["x_u8"], dtype=np.uint8)
        bits = np.array([case["bits_word_with_tail_garbage"]], dtype=np.uint32)
        for sp, fmt in ((x, "u8"), (bits, "bits")):
            acc, y = orc.project(Qc, s, N, K, sp, fmt, ldq=ldq)
            assert np.array_equal(acc[0], want_acc), (case["name"], fmt, acc)
            assert np.array_equal(f32_bits(y[0]), f32_bits(want_y)), (case["name"], fmt, y)
        if "y_sign_bits" in case:
            assert list((f32_bits(y[0]) >> 31).astype(int)) == case["y_sign_bits"]
        want_A = np.flatnonzero(x)
        assert np.array_equal(orc.active_set(x, "u8", K), want_A)
        assert np.array_equal(orc.active_set(bits, "bits", K), want_A)


def pin_exhaustive_small(orc):
    # N != K and ldq > N so a transposed operand or a dropped ldq shows.
    N, K, ldq = 5, 10, 7
    Qc, s, _ = synth.random_case(11, N, K, ldq=ldq)
    masks = ((np.arange(2 ** K)[:, None] >> np.arange(K)[None, :]) & 1).astype(np.uint8)
    acc, y = orc.project(Qc, s, N, K, masks, "u8", ldq=ldq)
    assert np.array_equal(acc.astype(np.int64), dense_ref(Qc, N, masks))
    acc_b, _ = orc.project(Qc, s, N, K, synth.pack_bits(masks), "bits", ldq=ldq)
    assert np.array_equal(acc_b, acc)


def pin_full_shapes(orc):
    for (N, K, p, seed) in ((1536, 1536, 0.1, 1), (1536, 6144, 0.2, 2),
                            (1536, 6144, 0.5, 3)):
        Qc, s, x = synth.random_case(seed, N, K, T=3, p=p)
        acc, y = orc.project(Qc, s, N, K, x, "u8")
        assert np.array_equal(acc.astype(np.int64), dense_ref(Qc, N, x))
        assert np.array_equal(f32_bits(y), f32_bits(exact_scaled(acc, s[None, :])))


def pin_scale_rounding(orc):
    N, K = 64, 300
    rng = synth.rng_for(77)
    Qc = rng.integers(-128, 128, size=(K, N)).astype(np.int8)
    # scales with full 24-bit significands over a wide exponent range, both signs
    s = (rng.uniform(1, 2, N) * 2.0 ** rng.integers(-30, 30, N)
         * rng.choice([-1.0, 1.0], N)).astype(np.float32)
    x = synth.bernoulli(rng, (4, K), 0.6)
    x[0] = 0                          # zero sums: signed zeros
    acc, y = orc.project(Qc, s, N, K, x, "u8")
    assert np.array_equal(f32_bits(y), f32_bits(exact_scaled(acc, s[None, :])))
    assert np.all((f32_bits(y[0]) >> 31) == (f32_bits(s) >> 31))


def pin_invariants(orc):
    N, K, ldq = 48, 200, 64
    Qc, s, x = synth.random_case(5, N, K, T=2, p=0.3, ldq=ldq)
    L = logical(Qc, N)
    # zero spikes -> zero accumulators
    acc0, _ = orc.project(Qc, s, N, K, np.zeros(K, np.uint8), "u8", ldq=ldq)
    assert not acc0.any()
    # one-hot e_k -> column k and y = s * float(column)
    for k in (0, 1, 31, 32, 100, K - 1):
        e = np.zeros(K, np.uint8)
        e[k] = 1
        acc, y = orc.project(Qc, s, N, K, e, "u8", ldq=ldq)
        assert np.array_equal(acc[0], L[:, k]), k
        assert np.array_equal(f32_bits(y[0]), f32_bits(s * L[:, k].astype(np.float32)))
    # additivity over disjoint active sets
    a = x[0] & (np.arange(K) % 2 == 0)
    b = x[1] & (np.arange(K) % 2 == 1)
    acc_ab, _ = orc.project(Qc, s, N, K, (a | b)[None], "u8", ldq=ldq)
    acc_a, _ = orc.project(Qc, s, N, K, a[None], "u8", ldq=ldq)
    acc_b, _ = orc.project(Qc, s, N, K, b[None], "u8", ldq=ldq)
    assert np.array_equal(acc_ab, acc_a + acc_b)
    # all ones -> row sums
    acc1, _ = orc.project(Qc, s, N, K, np.ones(K, np.uint8), "u8", ldq=ldq)
    assert np.array_equal(acc1[0], L.sum(axis=1))
    # permuting columns of Q together with x changes nothing
    perm = synth.rng_for(6).permutation(K)
    accp, _ = orc.project(np.ascontiguousarray(Qc[perm]), s, N, K, x[:, perm], "u8", ldq=ldq)
    accx, yx = orc.project(Qc, s, N, K, x, "u8", ldq=ldq)
    assert np.array_equal(accp, accx)
    # bits == u8; tail bits past K ignored; any nonzero byte is a spike
    bits = synth.pack_bits(x)
    bits[:, -1] |= np.uint32(0xFFFFFFFF) << np.uint32(K % 32)
    accb, yb = orc.project(Qc, s, N, K, bits, "bits", ldq=ldq)
    assert np.array_equal(accb, accx) and np.array_equal(f32_bits(yb), f32_bits(yx))
    xv = x * synth.rng_for(8).integers(1, 256, size=x.shape).astype(np.uint8)
    accv, _ = orc.project(Qc, s, N, K, xv, "u8", ldq=ldq)
    assert np.array_equal(accv, accx)
    # rows are independent: a batch equals its rows one at a time
    for t in range(x.shape[0]):
        acct, _ = orc.project(Qc, s, N, K, x[t], "u8", ldq=ldq)
        assert np.array_equal(acct[0], accx[t])
    # active set is the ascending list of firing columns
    assert np.array_equal(orc.active_set(x[0], "u8", K), np.flatnonzero(x[0]))
    assert np.array_equal(orc.active_set(bits[0], "bits", K), np.flatnonzero(x[0]))


def pin_closed_forms(orc):
    N, K = 32, 4096
    x = synth.bernoulli(synth.rng_for(9), (3, K), 0.25)
    x[2] = 1
    nA = x.astype(np.int64).sum(axis=1)
    s = np.ones(N, np.float32)
    for c in (1, -1, 127, -127, -128, 0, 5):
        Qc = np.full((K, N), c, dtype=np.int8)
        acc, y = orc.project(Qc, s, N, K, x, "u8")
        assert np.array_equal(acc, np.repeat((c * nA)[:, None], N, 1).astype(np.int32)), c
        assert np.array_equal(y, acc.astype(np.float32))


def pin_overflow_reported(orc):
    # -128 * (2^24 + 1) = -2^31 - 128 does not fit INT32: must be an error,
    # never a wrapped value.
    K = (1 << 24) + 1
    Qc = np.full((K, 1), -128, dtype=np.int8)
    x = np.ones(K, np.uint8)
    try:
        orc.project(Qc, np.ones(1, np.float32), 1, K, x, "u8")
    except RuntimeError:
        pass
    else:
        raise AssertionError("INT32 overflow not reported")
    # the largest sum that fits is exact
    K2 = (1 << 24)
    acc, _ = orc.project(Qc[:K2], np.ones(1, np.float32), 1, K2, x[:K2], "u8")
    assert acc[0, 0] == -(1 << 31)


def pin_entries(orc):
    N, K, T = 96, 333, 5
    Qc, s, x = synth.random_case(12, N, K, T=T, p=0.2, ldq=112)
    acc, y = orc.project(Qc, s, N, K, x, "u8", ldq=112)
    rng = synth.rng_for(13)
    t = rng.integers(0, T, 200)
    m = rng.integers(0, N, 200)
    ae, ye = orc.project_entries(Qc, s, N, K, x, "u8", t, m, ldq=112)
    assert np.array_equal(ae, acc[t, m])
    assert np.array_equal(f32_bits(ye), f32_bits(y[t, m]))
    be, _ = orc.project_entries(Qc, s, N, K, synth.pack_bits(x), "bits", t, m, ldq=112)
    assert np.array_equal(be, ae)


# --- continuous-input projection ---------------------------------------------

def dense_case(seed, N, K, T, ldq, ldx):
    """Row-major Q [N, ldq] with random padding, x float32 [T, ldx] whose
    columns past K are large (so a read past K shows), scale [N]."""
    rng = synth.rng_for(300 + seed, N, K, T)
    Q = rng.integers(-128, 128, size=(N, ldq)).astype(np.int8)
    x = rng.standard_normal((T, ldx)).astype(np.float32)
    x[:, K:] = 1.0e6
    s = rng.uniform(0.25, 2.0, N).astype(np.float32)
    return Q, x, s


def pin_dense_hand_fixture(orc):
    g = json.loads((GOLDEN / "hand_worked_dense.json").read_text())
    Q = np.array(g["Q_rows"], np.int8)
    y, mag = orc.dense(Q, np.array(g["s"], np.float32), g["N"], g["K"],
                       np.array(g["x"], np.float32), ldq=g["ldq"])
    assert y[0].tolist() == g["y"], (y, g["y"])
    assert mag[0].tolist() == g["abs_dot"], (mag, g["abs_dot"])


def pin_dense_matmul(orc):
    # N != K, ldq > K and ldx > K so a transposed operand, a dropped stride
    # or a read past K shows.
    for (N, K, T, ldq, ldx, seed) in ((7, 13, 3, 16, 20, 1), (64, 300, 2, 304, 308, 2),
                                      (1536, 1536, 1, 1536, 1540, 3)):
        Q, x, s = dense_case(seed, N, K, T, ldq, ldx)
        y, mag = orc.dense(Q, s, N, K, x, ldq=ldq)
        Ql = Q[:, :K].astype(np.float64)
        xl = x[:, :K].astype(np.float64)
        want = (xl @ Ql.T) * s.astype(np.float64)[None, :]
        want_mag = np.abs(xl) @ np.abs(Ql).T
        tol = 4 * K * 2.0 ** -53 * want_mag * s.astype(np.float64)[None, :]
        assert np.all(np.abs(y - want) <= tol), np.max(np.abs(y - want) - tol)
        assert np.allclose(mag, want_mag, rtol=4 * K * 2.0 ** -53, atol=0)


def pin_dense_closed_forms(orc):
    N, K = 24, 1000
    s = np.linspace(0.5, 3.0, N).astype(np.float32)
    # constant Q = c, constant x = 0.5: every dot is c * K / 2 exactly
    for c in (1, -128, 127):
        Q = np.full((N, K), c, np.int8)
        y, _ = orc.dense(Q, s, N, K, np.full(K, 0.5, np.float32))
        assert np.array_equal(y[0], s.astype(np.float64) * (c * K / 2)), c
    Q, x, _ = dense_case(4, N, K, 1, K, K)
    # zero input, one-hot input (column k of Q times the scale)
    y, mag = orc.dense(Q, s, N, K, np.zeros(K, np.float32))
    assert not y.any() and not mag.any()
    for k in (0, 1, K // 2, K - 1):
        e = np.zeros(K, np.float32)
        e[k] = 1.0
        y, _ = orc.dense(Q, s, N, K, e)
        assert np.array_equal(y[0], s.astype(np.float64) * Q[:, k]), k


def pin_dense_linearity(orc):
    # dyadic inputs (multiples of 1/4, |x| <= 8): every partial sum is exact
    # in double, so y(x1 + x2) = y(x1) + y(x2) and y(-x) = -y(x) bit for bit
    N, K = 40, 257
    rng = synth.rng_for(305)
    Q = rng.integers(-128, 128, size=(N, K)).astype(np.int8)
    s = np.ones(N, np.float32)
    x1 = (rng.integers(-16, 17, K) / 4).astype(np.float32)
    x2 = (rng.integers(-16, 17, K) / 4).astype(np.float32)
    y1, _ = orc.dense(Q, s, N, K, x1)
    y2, _ = orc.dense(Q, s, N, K, x2)
    y12, _ = orc.dense(Q, s, N, K, x1 + x2)
    yn, _ = orc.dense(Q, s, N, K, -x1)
    assert np.array_equal(y12, y1 + y2)
    assert np.array_equal(yn, -y1)


def pin_dense_binary_is_sparse(orc):
    # for x in {0, 1}^K the dot product is the integer sum of Eq. (sparse)
    # over the active columns, and s * dot rounded to FP32 is the sparse y
    N, K, T = 48, 700, 4
    Q, _, s = dense_case(6, N, K, T, K, K)
    xb = synth.bernoulli(synth.rng_for(306), (T, K), 0.3)
    y, _ = orc.dense(Q, np.ones(N, np.float32), N, K, xb.astype(np.float32))
    acc, ysp = orc.project(np.ascontiguousarray(Q.T), s, N, K, xb, "u8")
    assert np.array_equal(y, acc.astype(np.float64))
    yd, _ = orc.dense(Q, s, N, K, xb.astype(np.float32))
    assert np.array_equal(yd.astype(np.float32), ysp)


# --- spike producer (LIF step) -------------------------------------------------

def rn32(q):
    """A rational rounded to the nearest float32, ties to even (exact)."""
    from fractions import Fraction
    f = np.float32(float(q))
    best = None
    for c in (np.nextafter(f, np.float32(-np.inf)), f, np.nextafter(f, np.float32(np.inf))):
        d = abs(Fraction(float(c)) - q)
        key = (d, int(np.array(c, np.float32).view(np.uint32)) & 1)
        if best is None or key < best[0]:
            best = (key, c)
    return np.float32(best[1])


def pin_lif_hand_fixture(orc):
    g = json.loads((GOLDEN / "hand_worked_lif.json").read_text())
    v, bits = orc.lif(np.array(g["v"], np.float32), np.array(g["I"], np.float32), g["K"],
                      g["beta"], g["theta"])
    assert v[0].tolist() == g["v_new"], v
    assert bits[0].tolist() == g["bits"], bits


def pin_lif_periodic(orc):
    # beta = 1/2, I = 1, theta = 7/4: v = 1, 3/2, 7/4 -> spike, 0, ... (all exact),
    # so every neuron fires on steps 2, 5, 8, ... and ends a step at v = 0 there
    K, T = 70, 3
    v = np.zeros((T, 72), np.float32)
    I = np.ones((T, 72), np.float32)
    v[:, K:] = 123.0                       # row padding: never touched
    for step in range(30):
        v, bits = orc.lif(v, I, K, 0.5, 1.75)
        fire = step % 3 == 2
        want = np.zeros(3, np.uint32)
        if fire:
            want[:] = [0xFFFFFFFF, 0xFFFFFFFF, (1 << 6) - 1]
        assert np.array_equal(bits, np.broadcast_to(want, (T, 3))), step
        assert np.all(v[:, :K] == [1.0, 1.5, 0.0][step % 3]), step
        assert np.all(v[:, K:] == 123.0)


def pin_lif_fma_rounding(orc):
    # beta * v + I with one rounding: exact rationals rounded once to FP32;
    # the inputs are chosen so that rounding the product first would differ
    from fractions import Fraction
    rng = synth.rng_for(310)
    cases = []
    while len(cases) < 16:
        b, v0, i0 = (np.float32(rng.uniform(0.5, 1.0)), np.float32(rng.normal()),
                     np.float32(rng.normal()))
        exact = Fraction(float(b)) * Fraction(float(v0)) + Fraction(float(i0))
        if rn32(exact) != np.float32(np.float32(b * v0) + i0):
            cases.append((b, v0, i0, rn32(exact)))
    for b, v0, i0, want in cases:
        v, bits = orc.lif(np.array([v0], np.float32), np.array([i0], np.float32), 1, float(b),
                          float("inf"))
        assert v[0, 0] == want and bits[0, 0] == 0, (b, v0, i0, v[0, 0], want)


def pin_lif_bits_format(orc):
    # dyadic inputs: beta * v + I is exact, so the spikes are known; the bits
    # must unpack (through the spike oracle) to exactly those columns, and the
    # words past K must be zero
    K = 83
    rng = synth.rng_for(311)
    v = (rng.integers(-64, 64, (4, K)) / 32).astype(np.float32)
    I = (rng.integers(-64, 64, (4, K)) / 32).astype(np.float32)
    pre = 0.75 * v.astype(np.float64) + I.astype(np.float64)
    vn, bits = orc.lif(v, I, K, 0.75, 0.5)
    for t in range(4):
        fired = np.flatnonzero(pre[t] >= 0.5)
        assert np.array_equal(orc.active_set(bits[t], "bits", K), fired), t
        assert (int(bits[t, -1]) >> (K % 32)) == 0, "tail bits set"
        want_v = np.where(pre[t] >= 0.5, pre[t] - 0.5, pre[t]).astype(np.float32)
        assert np.array_equal(vn[t], want_v), t
    # an infinite threshold never fires
    _, bits = orc.lif(v, I, K, 0.75, float("inf"))
    assert not bits.any()


def _head_case(seed, V, K, B=1, ldq_pad=0, ldh_pad=0):
    rng = synth.rng_for(7700, seed, V, K, B)
    Q = rng.integers(-127, 128, size=(V, K + ldq_pad)).astype(np.int8)
    s = rng.uniform(0.01, 0.05, size=V).astype(np.float32)
    h = rng.standard_normal((B, K + ldh_pad)).astype(np.float32)
    return Q, s, h


def pin_head_hand_fixture(orc):
    g = json.loads((GOLDEN / "hand_worked_head.json").read_text())
    Q = np.array(g["Q_rows"], np.int8)
    s = np.array(g["s"], np.float32)
    h = np.array(g["h"], np.float32)
    for case in g["cases"]:
        o = orc.head(Q, s, g["V"], g["K"], h, case["tau"], case["k_sel"])
        assert o["codes"][0].tolist() == g["codes"]
        assert np.allclose(o["z"][0] / o["s_x"][0], g["z_over_s_x"], rtol=1e-6)
        assert np.isclose(o["s_x"][0], 2.0 / 127.0, rtol=1e-6)
        assert np.isclose(o["gap"][0], g["gap"], rtol=1e-5)
        assert int(o["verified"][0]) == case["verified"]
        assert o["cand"][0].tolist() == case["cand"]
        if "r" in case:
            assert np.allclose(o["r"][0], case["r"], rtol=1e-7)
        assert int(o["token"][0]) == case["token"]


def pin_head_integer_activations(orc):
    # h = q * 2^-4 with max |q| = 127: the scale is exactly 2^-4, the codes are
    # q, and the FP32-activation recompute (a separate loop over h) must equal
    # the approximate logit of the same row (both exact before one rounding)
    V, K, B = 40, 50, 2
    Q, s, _ = _head_case(1, V, K, B, ldq_pad=3)
    rng = synth.rng_for(7701)
    q = rng.integers(-127, 128, size=(B, K + 2)).astype(np.int64)
    q[:, 7] = 127
    q[1, 7] = -127
    h = (q * 2.0 ** -4).astype(np.float32)
    o = orc.head(Q, s, V, K, h, np.inf, V, ldq=K + 3)
    assert np.array_equal(o["codes"], q[:, :K].astype(np.int8))
    assert np.all(o["s_x"] == np.float32(2.0 ** -4))
    for b in range(B):
        assert np.array_equal(o["r"][b].astype(np.float32), o["z"][b][o["cand"][b]])
        # and both equal the integer product Q q (numpy int64) scaled
        a = Q[:, :K].astype(np.int64) @ q[b, :K]
        assert np.array_equal(o["r"][b], s[o["cand"][b]].astype(np.float64) * (a[o["cand"][b]] * 2.0 ** -4))


def pin_head_quantiser_rounding(orc):
    # with amax = 127 * 2^-3 the scale is exactly 2^-3: halves round to even
    K = 8
    h = (np.array([127, 2.5, -2.5, 3.5, 0.5, -0.5, 1.5, 126.5]) * 2.0 ** -3).astype(np.float32)
    Q = np.ones((2, K), np.int8)
    o = orc.head(Q, np.ones(2, np.float32), 2, K, h, 0.0, 1)
    assert o["codes"][0].tolist() == [127, 2, -2, 4, 0, 0, 2, 126]
    assert o["s_x"][0] == np.float32(0.125)
    # below the 1e-8 floor the scale stays 1e-8 / 127 (about 7.874e-11)
    h = np.array([1e-10, -3e-9, 0.0], np.float32)
    o = orc.head(np.ones((2, 3), np.int8), np.ones(2, np.float32), 2, 3, h, 0.0, 1)
    assert o["codes"][0].tolist() == [1, -38, 0]
    assert np.isclose(o["s_x"][0], 1e-8 / 127, rtol=1e-6)


def pin_head_order_and_gate(orc):
    # duplicate rows give equal z: they must come in ascending index; the
    # order must be numpy's lexsort of (index, -z); the gate is strict
    V, K = 64, 33
    Q, s, h = _head_case(2, V, K)
    for dst, src in ((40, 3), (9, 3), (50, 61), (12, 61)):
        Q[dst], s[dst] = Q[src], s[src]
    o = orc.head(Q, s, V, K, h, 0.5, V)
    z = o["z"][0]
    assert z[9] == z[3] == z[40] and z[12] == z[50] == z[61]
    want = np.lexsort((np.arange(V), -z.astype(np.float64)))
    assert o["cand"][0].tolist() == want.tolist()
    g = np.float32(z[want[0]]) - np.float32(z[want[1]])
    assert o["gap"][0] == g
    for tau, want_v in ((0.0, 0), (float(g), 0), (float(np.nextafter(g, np.float32(np.inf))), 1),
                        (np.inf, 1)):
        assert int(orc.head(Q, s, V, K, h, tau, 4)["verified"][0]) == want_v, tau


def pin_head_permutation(orc):
    # renaming the rows renames the candidates and the token; permuting the
    # columns of Q and h together changes no decision
    V, K = 50, 40
    Q, s, h = _head_case(3, V, K)
    o = orc.head(Q, s, V, K, h, np.inf, 8)
    perm = synth.rng_for(7703).permutation(V)
    inv = np.argsort(perm)
    op = orc.head(Q[perm], s[perm], V, K, h, np.inf, 8)
    assert op["cand"][0].tolist() == inv[o["cand"][0]].tolist()
    assert int(op["token"][0]) == int(inv[o["token"][0]])
    cp = synth.rng_for(7704).permutation(K)
    oc = orc.head(Q[:, cp], s, V, K, h[:, cp], np.inf, 8)
    assert np.array_equal(oc["z"], o["z"]) and oc["cand"].tolist() == o["cand"].tolist()
    assert int(oc["token"][0]) == int(o["token"][0])
    assert np.allclose(oc["r"], o["r"], rtol=1e-12)


def pin_head_full_verification_is_dense_argmax(orc):
    # every row a candidate and the gate always open: the verified logits are
    # the continuous-input projection of h (the dense oracle), the token its
    # argmax; strides padded on both operands
    V, K, B = 45, 70, 2
    Q, s, h = _head_case(4, V, K, B, ldq_pad=5, ldh_pad=3)
    o = orc.head(Q, s, V, K, h, np.inf, V, ldq=K + 5)
    y, _ = orc.dense(Q, s, V, K, h, ldq=K + 5)
    for b in range(B):
        assert np.array_equal(o["r"][b], y[b][o["cand"][b]])
        assert int(o["token"][b]) == int(np.argmax(y[b]))


def pin_head_zero_state(orc):
    V, K = 10, 6
    Q, s, _ = _head_case(5, V, K)
    h = np.zeros(K, np.float32)
    o = orc.head(Q, s, V, K, h, 0.5, 4)
    assert np.all(o["codes"] == 0) and np.all(o["z"] == 0) and o["gap"][0] == 0
    assert int(o["verified"][0]) == 1 and o["cand"][0].tolist() == [0, 1, 2, 3]
    assert np.all(o["r"] == 0) and int(o["token"][0]) == 0
    o = orc.head(Q, s, V, K, h, 0.0, 4)
    assert int(o["verified"][0]) == 0 and int(o["token"][0]) == 0


ALL_PINS = [pin_hand_fixture, pin_exhaustive_small, pin_full_shapes,
            pin_scale_rounding, pin_invariants, pin_closed_forms,
            pin_overflow_reported, pin_entries,
            pin_dense_hand_fixture, pin_dense_matmul, pin_dense_closed_forms,
            pin_dense_linearity, pin_dense_binary_is_sparse,
            pin_lif_hand_fixture, pin_lif_periodic, pin_lif_fma_rounding, pin_lif_bits_format,
            pin_head_hand_fixture, pin_head_integer_activations, pin_head_quantiser_rounding,
            pin_head_order_and_gate, pin_head_permutation,
            pin_head_full_verification_is_dense_argmax, pin_head_zero_state]
