"""The allocation-free decode entry point (fixed static scratch, no plan)
against the plan-based spike_proj_decode and the CPU oracle, through the C
ABI.

The file name sorts last so that it also runs after every other test has
used the library in the same process; it passes alone as well."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth


def plan_decode(plan, spikes, fmt, N):
    acc = torch.full((N,), 7, dtype=torch.int32, device=DEV)
    y = torch.full((N,), 7.0, dtype=torch.float32, device=DEV)
    plan.decode(spikes, fmt, acc, y)
    return acc, y


def noalloc_decode(W, ldw, S, N, K, spikes, fmt):
    acc = torch.full((N,), -9, dtype=torch.int32, device=DEV)
    y = torch.full((N,), -9.0, dtype=torch.float32, device=DEV)
    sp.spike_proj_decode_noalloc(W, ldw, S, N, K, spikes, fmt, acc, y)
    return acc, y


@pytest.mark.gpu
@pytest.mark.parametrize("N,K,ldq,p", [
    (1536, 1536, 1536, 0.1),          # single projection, one chunk per tile
    (1536, 6144, 1536, 0.2),          # feed-forward down projection, split-K
    (2064, 1025, 2080, 0.5),          # ragged tile, ragged chunk, ldw > N
    (16, 1, 16, 1.0),                 # smallest shape
    (sp.SPIKE_PROJ_NOALLOC_MAX_N, 1100, sp.SPIKE_PROJ_NOALLOC_MAX_N, 0.3),  # largest N
    # K above 6144: split-K partials pass through the fixed scratch
    (2064, 8000, 2080, 0.2),
    (sp.SPIKE_PROJ_NOALLOC_MAX_N, 7000, sp.SPIKE_PROJ_NOALLOC_MAX_N, 0.1),
])
@pytest.mark.parametrize("fmt", ["bits", "u8"])
def test_noalloc_matches_plan_decode(N, K, ldq, p, fmt):
    Qc, s, x = synth.random_case(300 + K % 97, N, K, T=2, p=p, ldq=ldq)
    W, S = to_dev(Qc), to_dev(s)
    plan = sp.Plan(W, S, N, K, ldw=ldq)
    rows = to_dev(synth.pack_bits(x)) if fmt == "bits" else to_dev(x)
    ora_acc, ora_y = oracle.project(Qc, s, N, K, x, "u8", ldq=ldq)
    # two calls in a row on different spike rows: the second also shows that
    # the first left the shared scratch clean
    for t in range(2):
        want_acc, want_y = plan_decode(plan, rows[t], fmt, N)
        acc, y = noalloc_decode(W, ldq, S, N, K, rows[t], fmt)
        torch.cuda.synchronize()
        assert_parity(acc, y, want_acc.cpu().numpy(), want_y.cpu().numpy(),
                      f"N={N} K={K} {fmt} call {t} vs spike_proj_decode")
        assert_parity(acc, y, ora_acc[t], ora_y[t], f"N={N} K={K} {fmt} call {t} vs oracle")
    plan.close()


@pytest.mark.gpu
def test_noalloc_leaves_device_memory_alone():
    """After a first call, a few hundred more (split-K shapes included) leave
    the device's free memory exactly as it was: nothing is allocated."""
    cases = []
    for (N, K, ldq) in ((1536, 1536, 1536), (2064, 8000, 2080)):
        Qc, s, x = synth.random_case(400 + K, N, K, T=1, p=0.2, ldq=ldq)
        cases.append((to_dev(Qc), ldq, to_dev(s), N, K, to_dev(x[0]),
                      torch.empty(N, dtype=torch.int32, device=DEV),
                      torch.empty(N, dtype=torch.float32, device=DEV)))
    for (W, ldq, S, N, K, xr, acc, y) in cases:
        sp.spike_proj_decode_noalloc(W, ldq, S, N, K, xr, "u8", acc, y)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(200):
        for (W, ldq, S, N, K, xr, acc, y) in cases:
            sp.spike_proj_decode_noalloc(W, ldq, S, N, K, xr, "u8", acc, y)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


@pytest.mark.gpu
def test_noalloc_inside_graph_capture():
    """After the first call on the device, the entry point only enqueues its
    kernel, so it can be captured into a CUDA graph; replays give the
    oracle's results on whatever spike row the captured buffer holds."""
    N, K, ldq = 1536, 6144, 1536
    Qc, s, x = synth.random_case(451, N, K, T=3, p=0.15, ldq=ldq)
    W, S = to_dev(Qc), to_dev(s)
    rows = to_dev(x)
    row = rows[0].clone()
    acc = torch.empty(N, dtype=torch.int32, device=DEV)
    y = torch.empty(N, dtype=torch.float32, device=DEV)
    sp.spike_proj_decode_noalloc(W, ldq, S, N, K, row, "u8", acc, y)   # first call: outside capture
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        sp.spike_proj_decode_noalloc(W, ldq, S, N, K, row, "u8", acc, y,
                                     stream=torch.cuda.current_stream())
    want_acc, want_y = oracle.project(Qc, s, N, K, x, "u8", ldq=ldq)
    for t in (1, 2, 0):
        row.copy_(rows[t])
        g.replay()
        torch.cuda.synchronize()
        assert_parity(acc, y, want_acc[t], want_y[t], f"graph replay on row {t}")


@pytest.mark.gpu
def test_noalloc_rejects_n_above_the_scratch():
    N, K = sp.SPIKE_PROJ_NOALLOC_MAX_N + 16, 64
    W = torch.zeros((K, N), dtype=torch.int8, device=DEV)
    S = torch.ones(N, dtype=torch.float32, device=DEV)
    x = torch.ones(K, dtype=torch.uint8, device=DEV)
    acc = torch.zeros(N, dtype=torch.int32, device=DEV)
    with pytest.raises(sp.SpikeProjError) as e:
        sp.spike_proj_decode_noalloc(W, N, S, N, K, x, "u8", acc, None)
    assert e.value.status == sp.SP_ESCRATCH


def test_noalloc_size_check_on_the_host():
    """Too large an N is refused before any CUDA call (no GPU needed)."""
    from paper_2606_03026_gb300 import _build
    _build.build()
    fake = 1 << 20                       # never dereferenced: rejected first
    L = sp.lib()
    N = sp.SPIKE_PROJ_NOALLOC_MAX_N + 16
    assert L.spike_proj_decode_noalloc(fake, N, fake, N, 64, fake, 0, fake, None, None) == \
        sp.SP_ESCRATCH
    assert L.spike_proj_decode_noalloc(None, 16, fake, 16, 64, fake, 0, fake, None, None) == \
        sp.SP_EINVAL
    assert "scratch" in sp.spike_proj_strerror(sp.SP_ESCRATCH)
