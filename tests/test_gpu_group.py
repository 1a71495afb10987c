"""Grouped decode: the 44 binary-input projections of a 22-block decode step
in one launch, through the C ABI, against the CPU oracle (GPU)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def step():
    weights = synth.decode_step_weights(0)
    plans = [sp.Plan(to_dev(Q), to_dev(s), N, K) for (Q, s, N, K) in weights]
    group = sp.Group(plans)
    yield weights, plans, group
    group.close()


def step_inputs(weights, step_idx, p=0.1):
    Ks = [w[3] for w in weights]
    xs = synth.decode_step_spikes(step_idx, Ks, p=p)
    ld = (max(Ks) + 31) // 32
    bits = np.zeros((len(Ks), ld), np.uint32)
    u8 = np.zeros((len(Ks), max(Ks)), np.uint8)
    for j, x in enumerate(xs):
        b = synth.pack_bits(x)
        bits[j, : b.size] = b
        u8[j, : x.size] = x
    return xs, bits, u8


def oracle_step(weights, xs):
    accs, ys = [], []
    for (Q, s, N, K), x in zip(weights, xs):
        a, y = oracle.project(Q, s, N, K, x, "u8")
        accs.append(a[0])
        ys.append(y[0])
    return np.stack(accs), np.stack(ys)


@pytest.mark.parametrize("step_idx", [0, 1, 2])
def test_decode_step_22_blocks(step, step_idx):
    weights, plans, group = step
    xs, bits, u8 = step_inputs(weights, step_idx)
    want_acc, want_y = oracle_step(weights, xs)
    n = len(weights)
    acc = torch.full((n, 1536), -1, dtype=torch.int32, device=DEV)
    y = torch.full((n, 1536), -1.0, dtype=torch.float32, device=DEV)
    group.decode(to_dev(bits), "bits", bits.shape[1], acc, y, 1536)
    torch.cuda.synchronize()
    assert_parity(acc, y, want_acc, want_y, f"step {step_idx} bits")
    acc.fill_(0)
    y.fill_(0)
    group.decode(to_dev(u8), "u8", u8.shape[1], acc, y, 1536)
    torch.cuda.synchronize()
    assert_parity(acc, y, want_acc, want_y, f"step {step_idx} u8")
    assert group.status() == sp.SP_OK


def test_host_buffer_entry_point(step):
    """The host-buffer variant (copies inside the call) gives the same bits."""
    weights, plans, group = step
    xs, bits, _ = step_inputs(weights, 7)
    want_acc, want_y = oracle_step(weights, xs)
    n = len(weights)
    h_bits = torch.from_numpy(bits).pin_memory()
    h_acc = torch.empty((n, 1536), dtype=torch.int32).pin_memory()
    h_y = torch.empty((n, 1536), dtype=torch.float32).pin_memory()
    for _ in range(2):
        group.decode_host(h_bits, "bits", bits.shape[1], h_acc, h_y, 1536)
        torch.cuda.synchronize()
        assert_parity(h_acc, h_y, want_acc, want_y, "host buffers")


def test_host_buffer_pageable_and_page_locked(step):
    """Pageable host buffers go through device staging copies, page-locked
    ones are read and written in place by the kernel; both give the oracle's
    bits, with an output row stride wider than N."""
    weights, plans, group = step
    xs, bits, u8 = step_inputs(weights, 9)
    want_acc, want_y = oracle_step(weights, xs)
    n, ld = len(weights), 1600
    for locked in (False, True):
        for fmt, rows in (("bits", bits), ("u8", u8), ("bool8", u8 != 0)):
            h_rows = torch.from_numpy(np.ascontiguousarray(rows))
            h_acc = torch.full((n, ld), -3, dtype=torch.int32)
            h_y = torch.full((n, ld), -3.0, dtype=torch.float32)
            if locked:
                h_rows, h_acc, h_y = h_rows.pin_memory(), h_acc.pin_memory(), h_y.pin_memory()
            group.decode_host(h_rows, fmt, rows.shape[1], h_acc, h_y, ld)
            torch.cuda.synchronize()
            assert_parity(h_acc[:, :1536], h_y[:, :1536], want_acc, want_y,
                          f"host buffers locked={locked} {fmt}")
            assert (h_acc[:, 1536:] == -3).all() and (h_y[:, 1536:] == -3.0).all()


def test_mixed_group_shapes():
    """Projections of different N, K and ldw in one group, sparse and dense."""
    cases = [(16, 1), (48, 1000), (1552, 777), (512, 6144), (2048, 33)]
    weights, plans, xs = [], [], []
    for i, (N, K) in enumerate(cases):
        ldq = N + 16 * (i % 2)
        Qc, s, x = synth.random_case(40 + i, N, K, p=(0.05, 0.5, 1.0, 0.1, 0.0)[i], ldq=ldq)
        weights.append((Qc, s, N, K, ldq))
        plans.append(sp.Plan(to_dev(Qc), to_dev(s), N, K, ldw=ldq))
        xs.append(x[0])
    group = sp.Group(plans)
    maxK = max(K for _, K in cases)
    maxN = max(N for N, _ in cases)
    u8 = np.zeros((len(cases), maxK), np.uint8)
    for j, x in enumerate(xs):
        u8[j, : x.size] = x
    acc = torch.zeros((len(cases), maxN), dtype=torch.int32, device=DEV)
    y = torch.zeros((len(cases), maxN), dtype=torch.float32, device=DEV)
    group.decode(to_dev(u8), "u8", maxK, acc, y, maxN)
    torch.cuda.synchronize()
    for j, (Qc, s, N, K, ldq) in enumerate(weights):
        a, yy = oracle.project(Qc, s, N, K, xs[j], "u8", ldq=ldq)
        assert_parity(acc[j, :N], y[j, :N], a[0], yy[0], f"member {j}")
    group.close()


def test_group_of_64_uncached_masks():
    """The largest group (64 projections): 64 x 6144 columns of spike words
    exceed the shared-memory mask cache, so the kernel reads them from global
    memory; rates vary per member, some members have no spike at all."""
    N, K = 64, 6144
    weights, plans = [], []
    rng = synth.rng_for(99)
    rates = rng.uniform(0.0, 0.3, 64)
    rates[[3, 17, 40]] = 0.0
    X = (rng.random((64, K)) < rates[:, None]).astype(np.uint8)
    for j in range(64):
        Qc, s, _ = synth.random_case(200 + j, N, K, T=1)
        weights.append((Qc, s))
        plans.append(sp.Plan(to_dev(Qc), to_dev(s), N, K))
    group = sp.Group(plans)
    acc = torch.full((64, N), 3, dtype=torch.int32, device=DEV)
    y = torch.full((64, N), 3.0, dtype=torch.float32, device=DEV)
    bits = synth.pack_bits(X)
    group.decode(to_dev(bits), "bits", bits.shape[1], acc, y, N)
    torch.cuda.synchronize()
    for j, (Qc, s) in enumerate(weights):
        a, yy = oracle.project(Qc, s, N, K, X[j], "u8")
        assert_parity(acc[j], y[j], a[0], yy[0], f"member {j}")
    assert group.status() == sp.SP_OK
    group.close()


@pytest.mark.parametrize("p", [0.1, 1.0])
@pytest.mark.parametrize("ticket", [False, True])
def test_cluster_layouts(p, ticket):
    """Batch-1 groups run as clusters of 6 CTAs holding tiles x chunks:
    K <= 1024 (1 chunk, 6 tiles per cluster), <= 2048 (2 chunks, 3 tiles),
    <= 3072 (3 chunks, 2 tiles), <= 6144 (6 chunks, 1 tile), with tile counts
    that leave idle tile slots in the last cluster.  One member with K = 6145
    sends the whole group through the ticket form instead."""
    cases = [(2576, 1024), (1552, 1025), (2064, 2048), (1040, 2049), (1536, 3072),
             (528, 3073), (3088, 6144)] + ([(512, 6145)] if ticket else [])
    weights, plans, xs = [], [], []
    for i, (N, K) in enumerate(cases):
        Qc, s, x = synth.random_case(60 + i, N, K, p=p)
        weights.append((Qc, s, N, K))
        plans.append(sp.Plan(to_dev(Qc), to_dev(s), N, K))
        xs.append(x[0])
    group = sp.Group(plans)
    maxK = max(K for _, K in cases)
    maxN = max(N for N, _ in cases)
    bits = np.zeros((len(cases), (maxK + 31) // 32), np.uint32)
    for j, x in enumerate(xs):
        b = synth.pack_bits(x)
        bits[j, : b.size] = b
    for rep in range(2):
        acc = torch.full((len(cases), maxN), 5, dtype=torch.int32, device=DEV)
        y = torch.full((len(cases), maxN), 5.0, dtype=torch.float32, device=DEV)
        group.decode(to_dev(bits), "bits", bits.shape[1], acc, y, maxN)
        torch.cuda.synchronize()
        for j, (Qc, s, N, K) in enumerate(weights):
            a, yy = oracle.project(Qc, s, N, K, xs[j], "u8")
            assert_parity(acc[j, :N], y[j, :N], a[0], yy[0], f"member {j} rep {rep}")
            assert (acc[j, N:] == 5).all(), "wrote past the member's N"
    assert group.status() == sp.SP_OK
    group.close()


def test_large_mixed_group():
    """24 projections of 8 shapes in one launch (ragged N and K; 1, 3 and 6
    chunks per tile, so clusters of different layouts run side by side and
    more CTAs than SMs are resident), spike rates from 0 to 1.  Run twice:
    the second call must not see the first one's barriers."""
    shapes = [(1536, 6144), (1552, 1000), (512, 1024), (2064, 3073), (16, 1), (1040, 2049),
              (3088, 6144), (528, 200)]
    rates = [0.1, 0.05, 1.0, 0.1, 0.5, 0.0, 0.1, 0.3]
    cases = [(shapes[i % 8], rates[(i + i // 8) % 8]) for i in range(24)]

    weights, plans, xs = [], [], []
    for i, ((N, K), p) in enumerate(cases):
        Qc, s, x = synth.random_case(700 + i, N, K, p=p)
        weights.append((Qc, s, N, K))
        plans.append(sp.Plan(to_dev(Qc), to_dev(s), N, K))
        xs.append(x[0])
    group = sp.Group(plans)
    maxK = max(K for (_, K), _ in cases)
    maxN = max(N for (N, _), _ in cases)
    bits = np.zeros((len(cases), (maxK + 31) // 32), np.uint32)
    for j, x in enumerate(xs):
        b = synth.pack_bits(x)
        bits[j, : b.size] = b
    want = [oracle.project(Qc, s, N, K, x, "u8") for (Qc, s, N, K), x in zip(weights, xs)]
    for rep in range(2):
        acc = torch.full((len(cases), maxN), 5, dtype=torch.int32, device=DEV)
        y = torch.full((len(cases), maxN), 5.0, dtype=torch.float32, device=DEV)
        group.decode(to_dev(bits), "bits", bits.shape[1], acc, y, maxN)
        torch.cuda.synchronize()
        for j, (Qc, s, N, K) in enumerate(weights):
            assert_parity(acc[j, :N], y[j, :N], want[j][0][0], want[j][1][0], f"member {j} rep {rep}")
            assert (acc[j, N:] == 5).all(), "wrote past the member's N"
    assert group.status() == sp.SP_OK
    group.close()
