"""The device error word (failure detection without a GPU fault): a test
fault armed on a plan or group makes its next launch raise the error word and
stop half way -- outputs unwritten, split-K workspace and tile tickets left
dirty -- or, for the tensor-core kernel, makes one of its bounded waits run
out (~2 ms).  The status call must then report SP_EKERNEL once, clear the
word and re-zero the workspace, so that the next call is exact again against
the CPU oracle (GPU)."""
import time

import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu


def outputs(rows, N):
    return (torch.full((rows, N), -7, dtype=torch.int32, device=DEV),
            torch.full((rows, N), -7.0, dtype=torch.float32, device=DEV))


@pytest.fixture(scope="module")
def down():
    Qc, s = synth.down_weights(5)
    plan = sp.Plan(to_dev(Qc), to_dev(s), 1536, 6144, max_batch=512, gemm=True)
    yield Qc, s, plan
    plan.close()


def check_recovery(plan_or_group, call, want_acc, want_y, what, fault=sp.SP_FAULT_ABORT):
    """Arm the fault, run `call`, expect SP_EKERNEL once, then exact results."""
    acc, y = call()
    torch.cuda.synchronize()
    assert plan_or_group.status() == sp.SP_OK, f"{what}: error word set before the fault"
    plan_or_group.inject_fault(fault)
    t0 = time.perf_counter()
    acc, y = call()
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert dt < 5.0, f"{what}: the faulted launch took {dt:.2f} s"
    assert not np.array_equal(acc.cpu().numpy(), want_acc), f"{what}: output written anyway"
    assert plan_or_group.status() == sp.SP_EKERNEL, f"{what}: error word not raised"
    assert plan_or_group.status() == sp.SP_OK, f"{what}: error word not cleared"
    for rep in range(2):                   # the workspace and tickets were re-zeroed
        acc, y = call()
        torch.cuda.synchronize()
        assert_parity(acc, y, want_acc, want_y, f"{what}: call {rep} after recovery")
    assert plan_or_group.status() == sp.SP_OK


@pytest.mark.parametrize("strategy,T", [("gather", 5), ("gather", 64), ("union", 5), ("gemm", 5)])
def test_batched_abort(down, strategy, T):
    """The per-token gather at T = 5 rows (the cluster form: rows as a group
    of one-row problems) and T = 64 (more clusters than can be resident: the
    ticket form, 12 chunks per tile, workspace and tickets left dirty), the
    union fetch and the tensor-core GEMM, each stopped half way."""
    Qc, s, plan = down
    _, _, x = synth.random_case(17, 1536, 6144, T=T, p=0.15)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, x, "u8")
    xd = to_dev(x)

    def call():
        acc, y = outputs(T, 1536)
        plan.batched(xd, "u8", T, 6144, acc, y, strategy)
        return acc, y

    check_recovery(plan, call, want_acc, want_y, f"batched {strategy} T={T}")


def test_decode_abort(down):
    """Batch-1 decode (the cluster form, no workspace)."""
    Qc, s, plan = down
    _, _, x = synth.random_case(18, 1536, 6144, T=1, p=0.1)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, x, "u8")
    xd = to_dev(x[0])

    def call():
        acc, y = outputs(1, 1536)
        plan.decode(xd, "u8", acc[0], y[0])
        return acc, y

    check_recovery(plan, call, want_acc, want_y, "decode")


def test_decode_stall(down):
    """Batch-1 decode in clusters: the first CTA never stores its partial
    sums into the owners' shared memory, and the owners' bounded waits for
    them run out (about 2 ms under the stall fault)."""
    Qc, s, plan = down
    _, _, x = synth.random_case(20, 1536, 6144, T=1, p=0.1)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, x, "u8")
    xd = to_dev(x[0])

    def call():
        acc, y = outputs(1, 1536)
        plan.decode(xd, "u8", acc[0], y[0])
        return acc, y

    check_recovery(plan, call, want_acc, want_y, "decode stall", fault=sp.SP_FAULT_STALL)


def test_gemm_stall(down):
    """512-token prefill on the tensor cores (split-K clusters): one TMA copy
    is never issued and the MMA warp's bounded wait runs out; the kernel
    stops issuing, drains its copies, frees its tensor memory and returns."""
    Qc, s, plan = down
    X = synth.prefill_spikes(3)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, X, "u8")
    Xd = to_dev(X).bool()

    def call():
        acc, y = outputs(512, 1536)
        plan.batched(Xd, "bool8", 512, 6144, acc, y, "gemm")
        return acc, y

    check_recovery(plan, call, want_acc, want_y, "gemm stall", fault=sp.SP_FAULT_STALL)


def test_small_gemm_stall(down):
    """A few rows on the tensor cores (the small-T form, K split over a
    cluster): CTA 0's first weight box is never issued and its MMA thread's
    bounded wait runs out; it stores no partials, so the owners' bounded
    waits for them run out too."""
    Qc, s, plan = down
    _, _, x = synth.random_case(19, 1536, 6144, T=5, p=0.15)
    want_acc, want_y = oracle.project(Qc, s, 1536, 6144, x, "u8")
    xd = to_dev(x)

    def call():
        acc, y = outputs(5, 1536)
        plan.batched(xd, "u8", 5, 6144, acc, y, "gemm")
        return acc, y

    check_recovery(plan, call, want_acc, want_y, "small gemm stall", fault=sp.SP_FAULT_STALL)


def test_group_abort():
    """A decode step's group (ticket-free cluster form) at 3 and 22 blocks
    (the latter with more CTAs than SMs), aborted and stalled, and the
    grouped prefill (tail split: owners and helpers exchange partials behind
    flags)."""
    weights = synth.decode_step_weights(0, blocks=3)
    plans = [sp.Plan(to_dev(Q), to_dev(s), N, K, max_batch=256, gemm=True)
             for (Q, s, N, K) in weights]
    group = sp.Group(plans)
    Ks = [w[3] for w in weights]
    xs = synth.decode_step_spikes(7, Ks)
    u8 = np.zeros((len(Ks), max(Ks)), np.uint8)
    for j, x in enumerate(xs):
        u8[j, : x.size] = x
    want = [oracle.project(Q, s, N, K, x, "u8") for (Q, s, N, K), x in zip(weights, xs)]
    want_acc = np.concatenate([w[0] for w in want])
    want_y = np.concatenate([w[1] for w in want])
    u8d = to_dev(u8)

    def step():
        acc, y = outputs(len(Ks), 1536)
        group.decode(u8d, "u8", u8.shape[1], acc, y, 1536)
        return acc, y

    # the whole 22-block step
    wbig = synth.decode_step_weights(1)
    bplans = [sp.Plan(to_dev(Q), to_dev(s), N, K) for (Q, s, N, K) in wbig]
    big = sp.Group(bplans)
    bKs = [w[3] for w in wbig]
    bxs = synth.decode_step_spikes(8, bKs)
    bu8 = np.zeros((len(bKs), max(bKs)), np.uint8)
    for j, x in enumerate(bxs):
        bu8[j, : x.size] = x
    bwant = [oracle.project(Q, s, N, K, x, "u8") for (Q, s, N, K), x in zip(wbig, bxs)]
    want_big_acc = np.concatenate([w[0] for w in bwant])
    want_big_y = np.concatenate([w[1] for w in bwant])
    bu8d = to_dev(bu8)

    def big_step():
        acc, y = outputs(len(bKs), 1536)
        big.decode(bu8d, "u8", bu8.shape[1], acc, y, 1536)
        return acc, y

    check_recovery(group, step, want_acc, want_y, "group decode")
    check_recovery(big, big_step, want_big_acc, want_big_y, "group decode, 22 blocks")
    check_recovery(group, step, want_acc, want_y, "group decode stall", fault=sp.SP_FAULT_STALL)
    check_recovery(big, big_step, want_big_acc, want_big_y, "group decode stall, 22 blocks",
                   fault=sp.SP_FAULT_STALL)

    T = 256
    X = [synth.prefill_spikes(40 + j, T=T, K=K) for j, K in enumerate(Ks)]
    rows = [to_dev(np.pad(x, ((0, 0), (0, max(Ks) - x.shape[1])))).bool() for x in X]
    wantp = [oracle.project(Q, s, N, K, x, "u8") for (Q, s, N, K), x in zip(weights, X)]
    wantp_acc = np.stack([w[0] for w in wantp])
    wantp_y = np.stack([w[1] for w in wantp])

    def prefill():
        accs = [torch.full((T, 1536), -7, dtype=torch.int32, device=DEV) for _ in Ks]
        ys = [torch.full((T, 1536), -7.0, dtype=torch.float32, device=DEV) for _ in Ks]
        group.prefill(rows, "bool8", T, max(Ks), accs, ys)
        return torch.stack(accs), torch.stack(ys)

    check_recovery(group, prefill, wantp_acc, wantp_y, "group prefill")
    # the grouped prefill does not wait on other CTAs' copies: it ignores a
    # stall, which its launch still disarms
    group.inject_fault(sp.SP_FAULT_STALL)
    acc, y = prefill()
    torch.cuda.synchronize()
    assert_parity(acc, y, wantp_acc, wantp_y, "group prefill under an armed stall")
    assert group.status() == sp.SP_OK
    group.close()
    big.close()
    for p in plans + bplans:
        p.close()
