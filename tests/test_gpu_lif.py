"""Spike producer (spike_proj_lif) against the CPU oracle, bit for bit
(GPU): the membrane state and the BITS32 spike rows over many steps, ragged
K, padded rows, IEEE special values, and the produced rows fed straight into
the grouped decode step."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu


def lif_gpu(vd, Id, K, beta, theta, bits_d):
    rows, ld = vd.shape
    sp.spike_proj_lif(vd, Id, K, rows, ld, beta, theta, bits_d, bits_d.shape[1])
    torch.cuda.synchronize()


@pytest.mark.parametrize("K,rows", [(1, 1), (31, 3), (32, 2), (33, 5), (1000, 7), (6144, 44),
                                    (6161, 3)])
def test_lif_steps_bit_exact(K, rows):
    rng = synth.rng_for(820, K, rows)
    ld = K + 5
    words = (K + 31) // 32
    v = rng.normal(0.0, 1.0, (rows, ld)).astype(np.float32)
    v[:, K:] = 7.0                                     # row padding: never touched
    I = rng.normal(0.3, 1.0, (rows, ld)).astype(np.float32)
    vd, Id = to_dev(v), to_dev(I)
    bits_d = torch.full((rows, words + 2), 0x5A5A5A5A, dtype=torch.int32, device=DEV)
    for step in range(50):
        beta, theta = (0.9, 1.0) if step % 2 else (0.75, 0.5)
        v, want_bits = oracle.lif(v, I, K, beta, theta)
        lif_gpu(vd, Id, K, beta, theta, bits_d)
        got_v = vd.cpu().numpy()
        got_bits = bits_d.cpu().numpy().view(np.uint32)
        assert np.array_equal(got_v.view(np.uint32), v.view(np.uint32)), f"v differs at step {step}"
        assert np.array_equal(got_bits[:, :words], want_bits), f"bits differ at step {step}"
        assert np.all(got_bits[:, words:] == 0x5A5A5A5A), "wrote past ceil(K/32) words"


def test_lif_special_values():
    """Subnormal states stay subnormal (no flush to zero), NaN never fires
    and stays NaN (payloads are not compared), infinities behave as IEEE
    says, an exact threshold fires."""
    K = 12
    tiny = np.float32(1e-40)                           # subnormal
    v = np.array([[tiny, -tiny, np.nan, np.inf, -np.inf, 0.0, 1.0, 2.0, tiny, 0.5, -0.0, 3.0]],
                 np.float32)
    I = np.array([[0.0, 0.0, 1.0, 0.0, 5.0, tiny, 0.0, -1.0, tiny, 0.25, 0.0, np.nan]], np.float32)
    for beta, theta in ((1.0, 1.0), (0.5, 0.5), (1.0, -np.inf), (0.0, np.inf)):
        want_v, want_bits = oracle.lif(v, I, K, beta, theta)
        vd, Id = to_dev(v), to_dev(I)
        bits_d = torch.zeros((1, 1), dtype=torch.int32, device=DEV)
        lif_gpu(vd, Id, K, beta, theta, bits_d)
        got_v = vd.cpu().numpy()
        # bit for bit, except that a NaN is any NaN (the GPU returns its
        # canonical NaN, the CPU propagates the input's payload)
        both_nan = np.isnan(got_v) & np.isnan(want_v)
        assert np.array_equal(np.where(both_nan, 0, got_v.view(np.uint32)),
                              np.where(both_nan, 0, want_v.view(np.uint32))), (beta, theta, got_v, want_v)
        assert np.array_equal(bits_d.cpu().numpy().view(np.uint32), want_bits), (beta, theta)


def test_lif_feeds_group_decode():
    """The produced rows are the decode step's spike input as they stand:
    44 LIF layers (K = 1536 / 6144) -> spike_proj_group_decode equals the
    oracle projection of the oracle's spikes."""
    weights = synth.decode_step_weights(0, blocks=4)
    plans = [sp.Plan(to_dev(Q), to_dev(s), N, K) for (Q, s, N, K) in weights]
    group = sp.Group(plans)
    n, ld = len(weights), 6144
    words = ld // 32
    rng = synth.rng_for(821)
    v = rng.normal(0.0, 0.5, (n, ld)).astype(np.float32)
    I = rng.normal(0.1, 0.6, (n, ld)).astype(np.float32)
    vd, Id = to_dev(v), to_dev(I)
    bits_d = torch.zeros((n, words), dtype=torch.int32, device=DEV)
    acc = torch.empty((n, 1536), dtype=torch.int32, device=DEV)
    y = torch.empty((n, 1536), dtype=torch.float32, device=DEV)
    for step in range(3):
        v, want_bits = oracle.lif(v, I, ld, 0.8, 1.0)
        lif_gpu(vd, Id, ld, 0.8, 1.0, bits_d)
        group.decode(bits_d, "bits", words, acc, y, 1536)
        torch.cuda.synchronize()
        assert np.array_equal(bits_d.cpu().numpy().view(np.uint32), want_bits)
        for j, (Q, s, N, K) in enumerate(weights):
            wa, wy = oracle.project(Q, s, N, K, want_bits[j], "bits")
            assert_parity(acc[j], y[j], wa[0], wy[0], f"step {step} projection {j}")
