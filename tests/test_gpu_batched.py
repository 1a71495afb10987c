"""Batched decode and prefill: per-token gather, union shared fetch, the
tcgen05 tensor-core GEMM and the density dispatcher, all against the CPU
oracle and against each other (GPU)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu

STRATEGIES = ("gather", "union", "gemm")


def run_batched(plan, spikes, fmt, B, ld, N, strategy):
    acc = torch.full((B, N), -7, dtype=torch.int32, device=DEV)
    y = torch.full((B, N), -7.0, dtype=torch.float32, device=DEV)
    plan.batched(spikes, fmt, B, ld, acc, y, strategy)
    torch.cuda.synchronize()
    return acc, y


@pytest.fixture(scope="module")
def down():
    Qc, s = synth.down_weights(3)
    plan = sp.Plan(to_dev(Qc), to_dev(s), 1536, 6144, max_batch=512, gemm=True)
    return Qc, s, plan


@pytest.mark.parametrize("correlated", [False, True])
@pytest.mark.parametrize("strategy", STRATEGIES + ("auto",))
def test_batch64(down, correlated, strategy):
    """B = 64 tokens, rates U(0.05, 0.2), independent or hot-set correlated."""
    Qc, s, plan = down
    X, _, _ = synth.batched_spikes(0, correlated=correlated)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, X, "u8")
    bits = synth.pack_bits(X)
    acc, y = run_batched(plan, to_dev(bits), "bits", 64, bits.shape[1], 1536, strategy)
    assert_parity(acc, y, want_acc, want_y, f"B=64 {strategy} corr={correlated}")
    for fmt in ("u8", "bool8"):
        acc, y = run_batched(plan, to_dev(X), fmt, 64, X.shape[1], 1536, strategy)
        assert_parity(acc, y, want_acc, want_y, f"B=64 {fmt} {strategy} corr={correlated}")
    if strategy == "auto":
        chosen, active = plan.last_dispatch()
        assert chosen in STRATEGIES
        assert active == int(X.astype(np.int64).sum())


def test_prefill_512_tokens(down):
    """512-token prefill block: X ~ Bernoulli(0.15 * lognormal(0, 0.5)); the
    dispatcher must pick the tensor-core GEMM; full output vs the oracle."""
    Qc, s, plan = down
    X = synth.prefill_spikes(0)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, X, "u8")
    Xd = to_dev(X)
    acc = torch.empty(512, 1536, dtype=torch.int32, device=DEV)
    y = torch.empty(512, 1536, dtype=torch.float32, device=DEV)
    plan.prefill(Xd, 512, 6144, acc, y, "auto")
    torch.cuda.synchronize()
    assert plan.last_dispatch() == ("gemm", int(X.astype(np.int64).sum()))
    assert_parity(acc, y, want_acc, want_y, "prefill auto")
    for strategy in ("gemm", "gather", "union"):
        acc.fill_(0)
        y.fill_(0)
        plan.prefill(Xd, 512, 6144, acc, y, strategy)
        torch.cuda.synchronize()
        assert_parity(acc, y, want_acc, want_y, f"prefill {strategy}")
    # the same block as 0/1 bytes (a torch.bool tensor): read in place by the GEMM
    Xbool = Xd.bool()
    acc, y = run_batched(plan, Xbool, "bool8", 512, 6144, 1536, "gemm")
    assert_parity(acc, y, want_acc, want_y, "prefill bool8 in place")
    assert plan.status() == sp.SP_OK


@pytest.mark.parametrize("T,N,K,ldq", [(1, 16, 1, 16), (5, 48, 100, 64), (129, 272, 1000, 288),
                                       (300, 1552, 777, 1552), (128, 256, 64, 256),
                                       (257, 512, 6143, 512)])
def test_gemm_ragged(T, N, K, ldq):
    """The tensor-core path on ragged row / column / K-block tails."""
    Qc, s, X = synth.random_case(60 + T, N, K, T=T, p=0.3, ldq=ldq)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8", ldq=ldq)
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, ldw=ldq, max_batch=T, gemm=True)
    for strategy in STRATEGIES:
        acc, y = run_batched(plan, to_dev(X), "u8", T, K, N, strategy)
        assert_parity(acc, y, want_acc, want_y, f"T={T} N={N} K={K} {strategy}")


@pytest.mark.parametrize("T,N,K", [(1, 16, 1), (5, 48, 100), (129, 272, 1000), (300, 1552, 777),
                                   (257, 512, 6143)])
def test_gemm_u8_rows_any_nonzero(T, N, K):
    """u8 spike rows on the tensor-core path: any nonzero byte is a spike
    (the 0/1 staging pass maps them), bytes past K in each row are ignored,
    rows and K-blocks ragged."""
    Qc, s, X = synth.random_case(80 + T, N, K, T=T, p=0.3)
    ldx = (K + 15) // 16 * 16 + 16
    rng = synth.rng_for(81, T, K)
    Xs = rng.integers(1, 256, size=(T, ldx)).astype(np.uint8)     # garbage past K
    Xs[:, :K] = np.where(X != 0, rng.integers(1, 256, size=(T, K)), 0).astype(np.uint8)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=T, gemm=True)
    for rep in range(2):
        acc, y = run_batched(plan, to_dev(Xs), "u8", T, ldx, N, "gemm")
        assert_parity(acc, y, want_acc, want_y, f"T={T} N={N} K={K} rep {rep}")
    assert plan.status() == sp.SP_OK


@pytest.mark.parametrize("T,N,K", [(1, 16, 1), (5, 48, 100), (129, 272, 1000), (300, 1552, 777),
                                   (257, 512, 6143), (512, 1536, 6144)])
def test_gemm_bool8_rows(T, N, K):
    """0/1 byte rows (SP_SPIKES_BOOL8): with a 16-byte-aligned row stride the
    tensor-core kernel reads them in place (bytes past K ignored, whatever
    they hold); with an odd stride they go through the staging pass.  Both
    equal the oracle and the gather path bit for bit."""
    Qc, s, X = synth.random_case(90 + T, N, K, T=T, p=0.3)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=T, gemm=True)
    rng = synth.rng_for(91, T, K)
    for ldx in ((K + 15) // 16 * 16 + 16, K + 1 if (K + 1) % 16 else K + 2):
        Xs = rng.integers(2, 256, size=(T, ldx)).astype(np.uint8)    # not 0/1 past K
        Xs[:, :K] = X != 0
        Xd = to_dev(Xs)
        for strategy in ("gemm", "gemm", "gather"):
            acc, y = run_batched(plan, Xd, "bool8", T, ldx, N, strategy)
            assert_parity(acc, y, want_acc, want_y, f"T={T} N={N} K={K} ldx={ldx} {strategy}")
    assert plan.status() == sp.SP_OK


@pytest.mark.parametrize("T,N,K", [(2, 1536, 6144), (5, 272, 1000), (17, 1552, 777), (33, 1536, 6144),
                                   (64, 528, 3073), (65, 1040, 2049), (3, 2064, 8000), (9, 16, 1)])
def test_gather_rows(T, N, K):
    """The gather strategy on T rows: up to 64 rows run as a group of
    one-row problems (the cluster form when every cluster fits at once, else
    the ticket form with the batched form's workspace offsets; K above 6144
    is always the ticket form), more than 64 in the batched ticket form.
    Rows of mixed rates, every format, twice in a row (the second call must
    find the workspace and tickets clean)."""
    rng = synth.rng_for(95, T, N, K)
    Qc, s, _ = synth.random_case(96 + T, N, K, T=1)
    rates = rng.uniform(0.0, 0.4, size=(T, 1))
    rates[0] = 1.0
    X = (rng.random((T, K)) < rates).astype(np.uint8)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=T)
    bits = synth.pack_bits(X)
    for rep in range(2):
        for fmt, rows, ld in (("bits", bits, bits.shape[1]), ("u8", X, K)):
            acc, y = run_batched(plan, to_dev(rows), fmt, T, ld, N, "gather")
            assert_parity(acc, y, want_acc, want_y, f"T={T} N={N} K={K} {fmt} rep {rep}")
    assert plan.status() == sp.SP_OK
    plan.close()


def test_gemm_extremes():
    """All-ones spikes against -128 / +127 weights: the largest sums the
    tensor-core path must carry exactly (|acc| = 128 * K)."""
    T, N, K = 130, 64, 8192
    X = np.ones((T, K), np.uint8)
    X[1::2, ::3] = 0
    s = np.linspace(-2, 2, N).astype(np.float32)
    for c, other in ((-128, 127), (127, -127), (127, 1), (-128, -1)):
        Qc = np.full((K, N), c, np.int8)
        Qc[::5] = other                  # (127, 1) and (-128, -1): large odd sums
        want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
        plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=T, gemm=True)
        for fmt in ("u8", "bool8"):
            acc, y = run_batched(plan, to_dev(X), fmt, T, K, N, "gemm")
            assert_parity(acc, y, want_acc, want_y, f"gemm extremes {c} {other} {fmt}")


def test_gemm_largest_k():
    """K = SPIKE_PROJ_MAX_K on the tensor-core path: all-ones spikes against
    -128 weights give acc = -2^24 exactly (the exactness boundary), and
    +127 / +1 mixes give large odd sums; K is split 8 ways here."""
    T, N, K = 130, 64, sp.SPIKE_PROJ_MAX_K
    X = np.ones((T, K), np.uint8)
    X[1::2, ::7] = 0
    s = np.linspace(-1, 1, N).astype(np.float32)
    for c, other in ((-128, -128), (127, 1)):
        Qc = np.full((K, N), c, np.int8)
        Qc[::3] = other
        want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
        if c == -128:
            assert int(want_acc[0, 0]) == -(1 << 24)
        plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=T, gemm=True)
        for fmt in ("bool8", "u8"):
            acc, y = run_batched(plan, to_dev(X), fmt, T, K, N, "gemm")
            assert_parity(acc, y, want_acc, want_y, f"gemm K max {c} {fmt}")
        assert plan.status() == sp.SP_OK
        plan.close()


def test_auto_dispatch_by_cost(down):
    """SP_AUTO: per-token gather for small batches, the tensor-core GEMM for
    large ones on a plan with SP_PLAN_GEMM, never the GEMM without it; the
    result is the same bits either way."""
    Qc, s, plan = down
    X = np.concatenate([synth.batched_spikes(i)[0] for i in range(4)])        # 256 tokens
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, X, "u8")
    bits = to_dev(synth.pack_bits(X))
    for B, expect in ((8, "gather"), (256, "gemm")):
        acc, y = run_batched(plan, bits, "bits", B, bits.shape[1], 1536, "auto")
        assert plan.last_dispatch()[0] == expect, (B, plan.last_dispatch())
        assert_parity(acc, y, want_acc[:B], want_y[:B], f"auto B={B}")
    plain = sp.Plan(to_dev(Qc), to_dev(s), 1536, 6144, max_batch=256)
    acc, y = run_batched(plain, bits, "bits", 256, bits.shape[1], 1536, "auto")
    assert plain.last_dispatch()[0] == "gather"
    assert_parity(acc, y, want_acc, want_y, "auto without the GEMM operand copy")
    plain.close()


def test_auto_dispatch_second_shape():
    """A 1536 x 1536 projection (the sequence-mixer shape): the small-T
    tensor-core form beats the gather at B = 16, one row and four rows stay
    on the gather (rows run as a group in the cluster form), and every
    choice is exact against the oracle."""
    c = synth.single_projection(4)
    Qc, s = c["Q"], c["s"]
    plan = sp.Plan(to_dev(Qc), to_dev(s), 1536, 1536, max_batch=64, gemm=True)
    rates = np.random.default_rng(5).uniform(0.05, 0.2, size=(64, 1))
    X = (np.random.default_rng(6).random((64, 1536)) < rates).astype(np.uint8)
    want_acc, want_y = oracle.project(Qc, s, 1536, 1536, X, "u8")
    bits = to_dev(synth.pack_bits(X))
    for B, expect in ((1, "gather"), (4, "gather"), (16, "gemm"), (64, "gemm")):
        acc, y = run_batched(plan, bits, "bits", B, bits.shape[1], 1536, "auto")
        assert plan.last_dispatch()[0] == expect, (B, plan.last_dispatch())
        assert_parity(acc, y, want_acc[:B], want_y[:B], f"1536 x 1536 auto B={B}")
    plan.close()


def test_union_many_rows():
    """More rows than one union launch holds (passes of 256)."""
    N, K, B = 256, 2000, 600
    Qc, s, X = synth.random_case(70, N, K, T=B, p=0.05)
    want_acc, want_y = oracle.project(Qc, s, N, K, X, "u8")
    plan = sp.Plan(to_dev(Qc), to_dev(s), N, K, max_batch=B)
    acc, y = run_batched(plan, to_dev(synth.pack_bits(X)), "bits", B, (K + 31) // 32, N, "union")
    assert_parity(acc, y, want_acc, want_y, "union 600 rows")


def test_errors_on_device():
    Qc, s, X = synth.random_case(80, 64, 128, T=4)
    W, S = to_dev(Qc), to_dev(s)
    plan = sp.Plan(W, S, 64, 128, max_batch=4)
    acc = torch.empty(8, 64, dtype=torch.int32, device=DEV)
    with pytest.raises(sp.SpikeProjError) as e:
        plan.batched(to_dev(X), "u8", 5, 128, acc, None, "gather")
    assert e.value.status == sp.SP_ERANGE
    with pytest.raises(sp.SpikeProjError) as e:
        plan.batched(to_dev(X), "u8", 4, 128, acc, None, "gemm")
    assert e.value.status == sp.SP_EUNSUPPORTED
    with pytest.raises(sp.SpikeProjError) as e:
        plan.batched(to_dev(X), "u8", 4, 100, acc, None, "gather")
    assert e.value.status == sp.SP_EINVAL
    with pytest.raises(sp.SpikeProjError) as e:
        plan.decode(to_dev(X[0]), "u8", None, None)
    assert e.value.status == sp.SP_EINVAL
    with pytest.raises(sp.SpikeProjError) as e:
        sp.Plan(W, S, 64, 128, ldw=72)
    assert e.value.status == sp.SP_EALIGN
    assert plan.status() == sp.SP_OK
