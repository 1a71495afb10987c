"""Batch-1 decode through the C ABI against the CPU oracle (GPU)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu


def run_decode(plan, spikes_dev, fmt, N):
    acc = torch.full((N,), 12345, dtype=torch.int32, device=DEV)
    y = torch.full((N,), 1.5, dtype=torch.float32, device=DEV)
    plan.decode(spikes_dev, fmt, acc, y)
    torch.cuda.synchronize()
    return acc, y


def test_single_projection_1536():
    """K = N = 1536, Bernoulli(0.1), uniform INT8, seed 0, both formats."""
    c = synth.single_projection(0)
    N, K = c["N"], c["K"]
    want_acc, want_y = oracle.project(c["Q"], c["s"], N, K, c["x"], "u8")
    plan = sp.Plan(to_dev(c["Q"]), to_dev(c["s"]), N, K)
    for fmt, x in (("u8", c["x"]), ("bool8", c["x"]), ("bits", c["bits"])):
        acc, y = run_decode(plan, to_dev(x), fmt, N)
        assert_parity(acc, y, want_acc[0], want_y[0], f"single {fmt}")
    assert plan.status() == sp.SP_OK


@pytest.mark.parametrize("p", synth.DOWN_RATES)
def test_down_projection_all_vectors(p):
    """K = 6144 -> N = 1536 at every spike rate: all 1000 seeded vectors per
    rate through the per-token gather (one launch), 20 of them also through
    single decode calls; every output checked against the oracle."""
    Qc, s = synth.down_weights(0)
    N, K = 1536, 6144
    X = synth.down_spikes(p, count=1000, seed=0)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
    W, S = to_dev(Qc), to_dev(s)
    plan = sp.Plan(W, S, N, K, max_batch=1000)
    bits = to_dev(synth.pack_bits(X))
    acc = torch.empty(1000, N, dtype=torch.int32, device=DEV)
    y = torch.empty(1000, N, dtype=torch.float32, device=DEV)
    plan.batched(bits, "bits", 1000, bits.shape[1], acc, y, "gather")
    torch.cuda.synchronize()
    assert_parity(acc, y, want_acc, want_y, f"down p={p}")
    Xd = to_dev(X)
    for t in range(0, 1000, 50):
        a1, y1 = run_decode(plan, Xd[t], "u8", N)
        assert_parity(a1, y1, want_acc[t], want_y[t], f"down p={p} t={t}")


@pytest.mark.parametrize("N,K,ldq", [(16, 1, 16), (16, 33, 32), (48, 1000, 64),
                                     (1552, 777, 1568), (528, 1025, 528), (512, 512, 512),
                                     (2048, 4096, 2048), (2064, 300, 2064), (4096, 2000, 4112),
                                     (6160, 129, 6160), (1536, 3000, 1536), (544, 2049, 560),
                                     (1040, 6145, 1040)])
@pytest.mark.parametrize("p", [0.0, 0.3, 1.0])
def test_ragged_shapes(N, K, ldq, p):
    """N not a multiple of the 512-channel tile, K with a ragged last word
    and chunk, ldw > N with random padding bytes, empty and full spike rows."""
    Qc, s, x = synth.random_case(7, N, K, T=2, p=p, ldq=ldq)
    want_acc, want_y = oracle.project(Qc, s, N, K, x, "u8", ldq=ldq)
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, ldw=ldq, max_batch=2)
    bits = synth.pack_bits(x)
    bits[:, -1] |= np.uint32(0xFFFFFFFF) << np.uint32(K % 32) if K % 32 else np.uint32(0)
    for t in range(2):
        acc, y = run_decode(plan, to_dev(bits[t]), "bits", N)
        assert_parity(acc, y, want_acc[t], want_y[t], f"N={N} K={K} bits t={t}")
        xv = x[t] * np.uint8(255)        # any nonzero byte is a spike
        acc, y = run_decode(plan, to_dev(xv), "u8", N)
        assert_parity(acc, y, want_acc[t], want_y[t], f"N={N} K={K} u8 t={t}")


# One shape for each cluster layout a single projection can take: (cluster
# size, chunks per tile) = (6, 1), (6, 2), (6, 6), (12, 3), (12, 6),
# (12, 12), (16, 1), (16, 2), (16, 4), (16, 8), (16, 16).  In each, every
# chunk's CTA stores its partial of each 4-channel group into the owning
# chunk's shared memory and the owner waits for kch x its groups' bytes.
@pytest.mark.parametrize("N,K", [(2576, 1), (1040, 600), (16, 1536), (2048, 768), (1040, 1536),
                                 (16, 3072), (6144, 1), (2576, 600), (1040, 1000), (1040, 2049),
                                 (16, 4100)])
def test_cluster_layouts_single(N, K):
    Qc, s, x = synth.random_case(900 + K % 101 + N % 7, N, K, T=2, p=0.3)
    x[1] = 1                                 # every column active: the largest sums
    want_acc, want_y = oracle.project(Qc, s, N, K, x, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K)
    bits = synth.pack_bits(x)
    for t in range(2):
        for fmt, rows in (("bits", bits), ("u8", x)):
            acc, y = run_decode(plan, to_dev(rows[t]), fmt, N)
            assert_parity(acc, y, want_acc[t], want_y[t], f"N={N} K={K} row {t} {fmt}")
    assert plan.status() == sp.SP_OK
    plan.close()


def test_one_hot_every_position():
    """e_k for every k of a ragged K: the output is column k times the scale."""
    N, K = 64, 300
    Qc, s, _ = synth.random_case(8, N, K)
    eye = np.eye(K, dtype=np.uint8)
    want_acc, want_y = oracle.project(Qc, s, N, K, eye, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=K)
    bits = to_dev(synth.pack_bits(eye))
    acc = torch.empty(K, N, dtype=torch.int32, device=DEV)
    y = torch.empty(K, N, dtype=torch.float32, device=DEV)
    plan.batched(bits, "bits", K, bits.shape[1], acc, y, "gather")
    torch.cuda.synchronize()
    assert_parity(acc, y, want_acc, want_y, "one-hot")
    assert np.array_equal(want_acc, Qc[:, :N].astype(np.int32))


def test_extremes_and_signed_zeros():
    """W = -128 / +127 everywhere at the largest K (|acc| reaches 2^24), zero
    and negative scales (signed zeros), and K = 131072."""
    N, K = 32, sp.SPIKE_PROJ_MAX_K
    x = np.ones(K, np.uint8)
    s = np.array([1.0, -1.0, 0.0, -0.0] * (N // 4), np.float32)
    for c in (-128, 127):
        Qc = np.full((K, N), c, np.int8)
        want_acc, want_y = oracle.project(Qc, s, N, K, x, "u8")
        assert abs(int(want_acc[0, 0])) == abs(c) * K
        plan = sp.Plan(to_dev(Qc), to_dev(s), N, K)
        acc, y = run_decode(plan, to_dev(synth.pack_bits(x)), "bits", N)
        assert_parity(acc, y, want_acc[0], want_y[0], f"extreme {c}")
    Qc = np.zeros((K, N), np.int8)
    acc, y = run_decode(sp.Plan(to_dev(Qc), to_dev(s), N, K), to_dev(x), "u8", N)
    yb = y.cpu().numpy().view(np.uint32)
    assert np.array_equal(yb >> 31, np.signbit(s).astype(np.uint32))


def test_repeatable_and_workspace_clean():
    """Repeated calls give identical bits (a race would show as a change) and
    leave no residue in the split-K workspace between calls."""
    Qc, s = synth.down_weights(1)
    N, K = 1536, 6144
    X = synth.down_spikes(0.2, count=3, seed=5)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K)
    Xd = to_dev(X)
    for rep in range(20):
        t = rep % 3
        acc, y = run_decode(plan, Xd[t], "u8", N)
        assert_parity(acc, y, want_acc[t], want_y[t], f"rep {rep}")
    assert plan.status() == sp.SP_OK


def test_acc_or_y_only():
    c = synth.single_projection(3)
    N, K = c["N"], c["K"]
    want_acc, want_y = oracle.project(c["Q"], c["s"], N, K, c["x"], "u8")
    plan = sp.Plan(to_dev(c["Q"]), to_dev(c["s"]), N, K)
    acc = torch.zeros(N, dtype=torch.int32, device=DEV)
    plan.decode(to_dev(c["bits"]), "bits", acc, None)
    y = torch.zeros(N, dtype=torch.float32, device=DEV)
    plan.decode(to_dev(c["bits"]), "bits", None, y)
    torch.cuda.synchronize()
    assert_parity(acc, y, want_acc[0], want_y[0], "split outputs")


def test_dense_long_rows_multi_round():
    """p = 0.95 over K = 100000 with N = 4096 (two output tiles, ~190k
    items): each CTA's share spans several rounds of the streaming kernel and
    tiles cross CTAs and rounds."""
    N, K = 4096, 100000
    Qc, s, x = synth.random_case(21, N, K, T=1, p=0.95)
    want_acc, want_y = oracle.project(Qc, s, N, K, x, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K)
    acc, y = run_decode(plan, to_dev(synth.pack_bits(x)[0]), "bits", N)
    assert_parity(acc, y, want_acc[0], want_y[0], "multi-round")
