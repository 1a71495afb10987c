"""The small-T tensor-core form (T <= 64 spike rows; Eq. (sparse) per token,
computed transposed with the output channels as the MMA's M and K split over
a cluster): bit-exact against the CPU oracle at the T boundaries, ragged N
and K, every input format, the largest sums, and the K limit of its
per-CTA spike slice, past which the launch falls back to the 128-row form
(GPU)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu


def run(plan, spikes, fmt, T, ld, N):
    acc = torch.full((T, N), -7, dtype=torch.int32, device=DEV)
    y = torch.full((T, N), -7.0, dtype=torch.float32, device=DEV)
    plan.batched(spikes, fmt, T, ld, acc, y, "gemm")
    torch.cuda.synchronize()
    return acc, y


@pytest.fixture(scope="module")
def down():
    Qc, s = synth.down_weights(9)
    plan = sp.Plan(to_dev(Qc), to_dev(s), 1536, 6144, max_batch=128, gemm=True)
    yield Qc, s, plan
    plan.close()


@pytest.mark.parametrize("T", [1, 2, 15, 16, 17, 33, 48, 63, 64, 65])
def test_down_projection_rows(down, T):
    """6144 -> 1536 at T around the 16-row MMA steps and the 64-row limit
    (65 takes the 128-row form); bits, u8 and bool8 rows, each twice (the
    second call must not see the first one's shared memory)."""
    Qc, s, plan = down
    rates = np.random.default_rng(T).uniform(0.05, 0.2, size=(T, 1))
    X = (np.random.default_rng(100 + T).random((T, 6144)) < rates).astype(np.uint8)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, X, "u8")
    bits = synth.pack_bits(X)
    for rep in range(2):
        acc, y = run(plan, to_dev(bits), "bits", T, bits.shape[1], 1536)
        assert_parity(acc, y, want_acc, want_y, f"T={T} bits rep {rep}")
    for fmt in ("u8", "bool8"):
        acc, y = run(plan, to_dev(X), fmt, T, 6144, 1536)
        assert_parity(acc, y, want_acc, want_y, f"T={T} {fmt}")
    assert plan.status() == sp.SP_OK


@pytest.mark.parametrize("T,N,K,ldq", [(17, 272, 1000, 288), (3, 16, 64, 16), (64, 400, 65, 400),
                                       (40, 1552, 777, 1552), (9, 128, 2049, 144)])
def test_ragged(T, N, K, ldq):
    """N not a multiple of the 128-channel tile, K not a multiple of the
    64-column K block (the tail of the last block is zero), ldw > N."""
    Qc, s, X = synth.random_case(300 + T, N, K, T=T, p=0.3, ldq=ldq)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8", ldq=ldq)
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, ldw=ldq, max_batch=T, gemm=True)
    bits = synth.pack_bits(X)
    acc, y = run(plan, to_dev(bits), "bits", T, bits.shape[1], N)
    assert_parity(acc, y, want_acc, want_y, f"T={T} N={N} K={K} bits")
    # u8 rows at an odd leading dimension (no 16-byte vector loads), any
    # nonzero byte a spike
    ldx = K + 3
    Xs = np.zeros((T, ldx), np.uint8)
    Xs[:, :K] = X * np.random.default_rng(T).integers(1, 256, size=X.shape)
    Xs[:, K:] = 9                        # past K: must be ignored
    acc, y = run(plan, to_dev(Xs), "u8", T, ldx, N)
    assert_parity(acc, y, want_acc, want_y, f"T={T} N={N} K={K} u8 ldx={ldx}")
    plan.close()


@pytest.mark.parametrize("K", [8192, 8193])
def test_extremes_at_the_k_limit(K):
    """All-ones rows against -128 / +127 weights: |acc| = 128 K, the largest
    sums.  K = 8192 is the longest K whose per-CTA spike slice fits (16 K
    blocks x 8 CTAs); K = 8193 falls back to the 128-row form."""
    T, N = 64, 128
    X = np.ones((T, K), np.uint8)
    X[1::2, ::3] = 0
    s = np.linspace(-2, 2, N).astype(np.float32)
    for c, other in ((-128, 127), (127, 1)):
        Qc = np.full((K, N), c, np.int8)
        Qc[::5] = other
        want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
        plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=T, gemm=True)
        for fmt in ("bool8", "u8"):
            acc, y = run(plan, to_dev(X), fmt, T, K, N)
            assert_parity(acc, y, want_acc, want_y, f"K={K} {c}/{other} {fmt}")
        assert plan.status() == sp.SP_OK
        plan.close()


def test_one_hot_rows(down):
    """Row t has the single spike k_t: acc row t is column k_t of W exactly,
    for k_t at the first, last and block-boundary columns."""
    Qc, s, plan = down
    ks = [0, 1, 63, 64, 767, 768, 4095, 6143]
    X = np.zeros((len(ks), 6144), np.uint8)
    for t, k in enumerate(ks):
        X[t, k] = 1
    acc, y = run(plan, to_dev(X), "u8", len(ks), 6144, 1536)
    want = np.stack([Qc[k].astype(np.int32) for k in ks])
    assert np.array_equal(acc.cpu().numpy(), want)
