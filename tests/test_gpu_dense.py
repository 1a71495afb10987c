"""Continuous-input projections (spike_proj_dense) against the CPU oracle
(GPU).  The kernel's FP32 result must lie within the error bound of its
fixed summation tree (depth d = 16 ceil(K / 512) + 5, see spike_proj.h) of
the oracle's near-exact double value; inputs whose every partial sum is
exact in FP32 (one-hot, 0/1 activations) must match bit for bit."""
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu

U = 2.0 ** -24


def tree_bound(K, s, mag, y_ref):
    """|y - y_exact| allowed for one output: gamma(d) |s| sum|W x| + 2u |y|."""
    d = 16 * math.ceil(K / 512) + 5
    g = d * U / (1 - d * U)
    return np.abs(s)[None, :] * g * mag + 2 * U * np.abs(y_ref) + 1e-45


def case(seed, N, K, B, ldw=None, ldx=None):
    rng = synth.rng_for(700 + seed, N, K, B)
    ldw = ldw or (K + 15) // 16 * 16
    ldx = ldx or (K + 3) // 4 * 4
    W = rng.integers(-128, 128, size=(N, ldw)).astype(np.int8)          # padding is random
    x = rng.standard_normal((B, ldx)).astype(np.float32)
    x[:, K:] = np.nan                                                   # must never be read
    s = rng.uniform(-2.0, 2.0, N).astype(np.float32)
    return W, x, s, ldw, ldx


def run(problems, B):
    """problems: list of (W, x, s, N, K, ldw, ldx); returns the y arrays."""
    keep, args, ys = [], [], []
    for (W, x, s, N, K, ldw, ldx) in problems:
        Wd, xd, sd = to_dev(W), to_dev(x), to_dev(s)
        y = torch.full((B, N + 3), float("nan"), dtype=torch.float32, device=DEV)
        keep += [Wd, xd, sd]
        ys.append(y)
        args.append((Wd, ldw, sd, xd, ldx, y, N + 3, N, K))
    sp.spike_proj_dense(args, B)
    torch.cuda.synchronize()
    out = [y.cpu().numpy() for y in ys]
    for y, (W, x, s, N, K, ldw, ldx) in zip(out, problems):
        assert np.isnan(y[:, N:]).all(), "wrote past N"
    return [y[:, :pr[3]] for y, pr in zip(out, problems)]


def check(y, W, x, s, N, K, ldw, what):
    want, mag = oracle.dense(W, s, N, K, x[:, :K], ldq=ldw)
    err = np.abs(y.astype(np.float64) - want)
    bound = tree_bound(K, s.astype(np.float64), mag, want)
    assert np.all(err <= bound), f"{what}: max excess {np.max(err - bound)}"


@pytest.mark.parametrize("N,K", [(1, 1), (5, 17), (33, 513), (100, 1000), (64, 1536),
                                 (7, 6144), (3, 6161)])
@pytest.mark.parametrize("B", [1, 2, 4])
def test_dense_vs_oracle(N, K, B):
    W, x, s, ldw, ldx = case(N + K, N, K, B, ldw=(K + 15) // 16 * 16 + 16, ldx=(K + 3) // 4 * 4 + 4)
    y, = run([(W, x, s, N, K, ldw, ldx)], B)
    check(y, W, x, s, N, K, ldw, f"N={N} K={K} B={B}")


def test_dense_largest_k():
    """K = SPIKE_PROJ_MAX_K (the tree is 16 * 256 + 5 deep) within its bound,
    and an exact case: constant weights and activations 1/4 (every partial
    sum a small dyadic multiple, exact in FP32)."""
    N, K, B = 9, sp.SPIKE_PROJ_MAX_K, 2
    W, x, s, ldw, ldx = case(77, N, K, B)
    y, = run([(W, x, s, N, K, ldw, ldx)], B)
    check(y, W, x, s, N, K, ldw, "K max")
    W = np.full((N, ldw), -3, np.int8)
    x = np.full((B, ldx), 0.25, np.float32)
    y, = run([(W, x, s, N, K, ldw, ldx)], B)
    assert np.array_equal(y, np.broadcast_to(s * np.float32(-0.75 * K), (B, N)))


def test_dense_group_mixed_shapes():
    """Many problems of different shapes in one launch (unit boundaries
    inside and across problems)."""
    shapes = [(1, 1), (4, 32), (5, 100), (9, 1536), (130, 777), (3, 4000), (64, 512), (17, 2049)]
    probs = []
    for i, (N, K) in enumerate(shapes * 3):
        W, x, s, ldw, ldx = case(40 + i, N, K, 3)
        probs.append((W, x, s, N, K, ldw, ldx))
    ys = run(probs, 3)
    for y, (W, x, s, N, K, ldw, ldx) in zip(ys, probs):
        check(y, W, x, s, N, K, ldw, f"group N={N} K={K}")


def test_dense_max_group():
    probs = []
    for i in range(sp.SPIKE_PROJ_DENSE_MAX_GROUP):
        W, x, s, ldw, ldx = case(200 + i, 8 + i % 5, 64 + 32 * (i % 7), 1)
        probs.append((W, x, s, W.shape[0], 64 + 32 * (i % 7), ldw, ldx))
    ys = run(probs, 1)
    for y, (W, x, s, N, K, ldw, ldx) in zip(ys, probs):
        check(y, W, x, s, N, K, ldw, "max group")


def test_dense_exact_cases():
    """One-hot activations give s_m * W[m][k] exactly; 0/1 activations give
    the spike-gated projection's y bit for bit (every partial sum is an
    integer below 2^24); zero activations give zero."""
    N, K, B = 300, 1536, 4
    W, _, s, ldw, ldx = case(9, N, K, B)
    x = np.zeros((B, ldx), np.float32)
    for b, k in enumerate((0, 17, 1023, K - 1)):
        x[b, k] = 1.0
    y, = run([(W, x, s, N, K, ldw, ldx)], B)
    for b, k in enumerate((0, 17, 1023, K - 1)):
        assert np.array_equal(y[b], s * W[:, k].astype(np.float32)), k
    xb = synth.bernoulli(synth.rng_for(710), (B, K), 0.3)
    x = np.zeros((B, ldx), np.float32)
    x[:, :K] = xb
    y, = run([(W, x, s, N, K, ldw, ldx)], B)
    _, ysp = oracle.project(np.ascontiguousarray(W[:, :K].T), s, N, K, xb, "u8")
    assert np.array_equal(y, ysp)
    y, = run([(W, np.zeros((B, ldx), np.float32), s, N, K, ldw, ldx)], B)
    assert not np.any(y)


def test_dense_decode_step_shapes_sampled():
    """The continuous projections of one block at full size (fused QKV 4608,
    attention output 1536, FFN up 6144 rows; K = 1536), one launch, checked
    on sampled rows against the oracle; and run-to-run bit identity."""
    probs = []
    for kind in ("qkv", "out", "up"):
        W, s = synth.dense_weights(0, kind)
        x = synth.hidden_state(0, B=1)
        probs.append((W, x, s, W.shape[0], W.shape[1], W.shape[1], W.shape[1]))
    ys = run(probs, 1)
    again = run(probs, 1)
    rng = synth.rng_for(711)
    for y, y2, (W, x, s, N, K, ldw, ldx) in zip(ys, again, probs):
        assert np.array_equal(y, y2), "not deterministic"
        rows = np.sort(rng.choice(N, 200, replace=False))
        want, mag = oracle.dense(np.ascontiguousarray(W[rows]), s[rows], len(rows), K, x, ldq=ldw)
        err = np.abs(y[:, rows].astype(np.float64) - want)
        assert np.all(err <= tree_bound(K, s[rows].astype(np.float64), mag, want))


def test_dense_errors():
    W = torch.zeros(16, 32, dtype=torch.int8, device=DEV)
    s = torch.ones(16, device=DEV)
    x = torch.ones(1, 32, device=DEV)
    y = torch.zeros(1, 16, device=DEV)
    good = (W, 32, s, x, 32, y, 16, 16, 32)
    bad = [((W, 8, s, x, 32, y, 16, 16, 32), sp.SP_EALIGN),      # ldw < K
           ((W, 32, s, x, 30, y, 16, 16, 32), sp.SP_EALIGN),     # ldx < K
           ((W, 32, s, x, 32, y, 8, 16, 32), sp.SP_EINVAL),      # ldy < N
           ((W, 32, s, x, 32, y, 16, 0, 32), sp.SP_EINVAL),      # N = 0
           ((W, 32, s, x, 32, y, 16, 16, sp.SPIKE_PROJ_MAX_K + 1), sp.SP_ERANGE)]
    for args, status in bad:
        with pytest.raises(sp.SpikeProjError) as e:
            sp.spike_proj_dense([args], 1)
        assert e.value.status == status, args
    with pytest.raises(sp.SpikeProjError):
        sp.spike_proj_dense([good], sp.SPIKE_PROJ_DENSE_MAX_B + 1)
    sp.spike_proj_dense([good], 1)
    torch.cuda.synchronize()
    assert torch.equal(y, torch.zeros_like(y))
