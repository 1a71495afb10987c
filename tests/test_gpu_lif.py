"""Spike producer (spike_proj_lif) against the CPU oracle, bit for bit
(GPU): the membrane state and the BITS32 spike rows over many steps, ragged
K, padded rows, IEEE special values, the produced rows fed straight into
the grouped decode step, and the producer fused into that step
(spike_proj_group_decode_lif, both of its forms)."""
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


@pytest.mark.parametrize("K,rows", [(1, 1), (31, 3), (32, 2), (33, 5), (127, 2), (129, 3),
                                    (1000, 7), (6144, 44), (6161, 3)])
@pytest.mark.parametrize("vector", [False, True])
def test_lif_steps_bit_exact(K, rows, vector):
    """ld = K + 5 takes the scalar form; ld a multiple of 4 (16-byte rows)
    the vector form once the state holds 2^22 neurons (rows are repeated to
    reach that size in the vector case)."""
    rng = synth.rng_for(820, K, rows)
    ld = (K + 3) // 4 * 4 + (4 if K % 4 == 0 else 0) if vector else K + 5
    if vector:
        rows = max(rows, -(-(1 << 22) // K))
        if rows * ld > (1 << 25):
            pytest.skip("vector case too large for the oracle here")
    words = (K + 31) // 32
    v = rng.normal(0.0, 1.0, (rows, ld)).astype(np.float32)
    v[:, K:] = 7.0                                     # row padding: never touched
    I = rng.normal(0.3, 1.0, (rows, ld)).astype(np.float32)
    vd, Id = to_dev(v), to_dev(I)
    bits_d = torch.full((rows, words + 2), 0x5A5A5A5A, dtype=torch.int32, device=DEV)
    for step in range(3 if vector else 50):
        beta, theta = (0.9, 1.0) if step % 2 else (0.75, 0.5)
        v, want_bits = oracle.lif(v, I, K, beta, theta)
        lif_gpu(vd, Id, K, beta, theta, bits_d)
        got_v = vd.cpu().numpy()
        got_bits = bits_d.cpu().numpy().view(np.uint32)
        assert np.array_equal(got_v.view(np.uint32), v.view(np.uint32)), f"v differs at step {step}"
        assert np.array_equal(got_bits[:, :words], want_bits), f"bits differ at step {step}"
        assert np.all(got_bits[:, words:] == 0x5A5A5A5A), "wrote past ceil(K/32) words"


def test_lif_large_state_vector():
    """The vector form on a 64-row x 65536-neuron state (the bench's stream
    shape, scaled down), several steps."""
    K, rows = 65536, 64
    rng = synth.rng_for(822)
    v = rng.normal(0.0, 1.0, (rows, K)).astype(np.float32)
    I = rng.normal(0.2, 0.8, (rows, K)).astype(np.float32)
    vd, Id = to_dev(v), to_dev(I)
    bits_d = torch.zeros((rows, K // 32), dtype=torch.int32, device=DEV)
    for step in range(3):
        v, want_bits = oracle.lif(v, I, K, 0.9, 1.0)
        lif_gpu(vd, Id, K, 0.9, 1.0, bits_d)
        assert np.array_equal(vd.cpu().numpy().view(np.uint32), v.view(np.uint32)), step
        assert np.array_equal(bits_d.cpu().numpy().view(np.uint32), want_bits), step


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


# ---------------------------------------------------------------------------
# the producer fused into the grouped decode (spike_proj_group_decode_lif)

def _fused_steps(weights, steps, with_bits, seed):
    """Runs `steps` fused decode steps, swapping the two state buffers, and
    checks every step against the oracle: the new state (bit for bit, rows
    past K_j untouched, the old state unchanged), the spike words and the
    projections."""
    plans = [sp.Plan(to_dev(Q), to_dev(s), N, K) for (Q, s, N, K) in weights]
    group = sp.Group(plans)
    n = len(weights)
    Ks = [w[3] for w in weights]
    maxK, maxN = max(Ks), max(w[2] for w in weights)
    ld = maxK + 3
    words = (maxK + 31) // 32
    rng = synth.rng_for(830, seed)
    v = rng.normal(0.0, 0.5, (n, ld)).astype(np.float32)
    for j, K in enumerate(Ks):
        v[j, K:] = 7.0
    bufs = [to_dev(v), torch.full((n, ld), 9.0, dtype=torch.float32, device=DEV)]
    pads = [v.copy(), np.full((n, ld), 9.0, np.float32)]
    bits_d = (torch.full((n, words + 1), 0x5A5A5A5A, dtype=torch.int32, device=DEV)
              if with_bits else None)
    acc = torch.empty((n, maxN), dtype=torch.int32, device=DEV)
    y = torch.empty((n, maxN), dtype=torch.float32, device=DEV)
    for step in range(steps):
        beta, theta = (0.9, 1.0) if step % 2 == 0 else (0.7, 0.6)
        I = rng.normal(0.15, 0.6, (n, ld)).astype(np.float32)
        vin, vout = bufs[step % 2], bufs[(step + 1) % 2]
        group.decode_lif(vin, vout, to_dev(I), beta, theta, bits=bits_d, acc=acc, y=y,
                         ld_out=maxN)
        torch.cuda.synchronize()
        got_in = vin.cpu().numpy()
        got_out = vout.cpu().numpy()
        assert np.array_equal(got_in.view(np.uint32), v.view(np.uint32)), f"v_in written, step {step}"
        new_v = v.copy()
        for j, (Q, s, N, K) in enumerate(weights):
            vj, bj = oracle.lif(v[j:j + 1], I[j:j + 1], K, beta, theta)
            new_v[j, :K] = vj[0, :K]
            assert np.array_equal(got_out[j, :K].view(np.uint32), vj[0, :K].view(np.uint32)), \
                f"step {step} state row {j}"
            pad = pads[(step + 1) % 2]
            assert np.array_equal(got_out[j, K:].view(np.uint32), pad[j, K:].view(np.uint32)), \
                f"step {step} row {j}: wrote past K"
            if with_bits:
                wj = (K + 31) // 32
                gb = bits_d[j].cpu().numpy().view(np.uint32)
                assert np.array_equal(gb[:wj], bj[0]), f"step {step} bits row {j}"
                assert np.all(gb[words:] == 0x5A5A5A5A), f"step {step} bits row {j} past ld"
            wa, wy = oracle.project(Q, s, N, K, bj[0], "bits", ldq=Q.shape[1])
            assert_parity(acc[j, :N], y[j, :N], wa[0], wy[0], f"step {step} projection {j}")
        # the buffer just written is the next step's input: its rows past K_j
        # keep their earlier contents
        v = new_v.copy()
        for j, K in enumerate(Ks):
            v[j, K:] = pads[(step + 1) % 2][j, K:]
    return group


def test_group_decode_lif_decode_step():
    """The 22-block decode step (44 projections, K = 1536 / 6144) with its
    spike producer fused in, three steps, spike words written out."""
    _fused_steps(synth.decode_step_weights(0), steps=3, with_bits=True, seed=1)


@pytest.mark.parametrize("with_bits", [True, False])
def test_group_decode_lif_ragged(with_bits):
    """Ragged N and K (chunk tails, a K below one word, partial tiles; N a
    multiple of 16 as plans require)."""
    shapes = [(16, 33), (496, 1000), (1536, 4097), (4000, 6144), (2096, 1536), (64, 32),
              (704, 6000), (16, 1)]
    weights = []
    for i, (N, K) in enumerate(shapes):
        Q, s, _ = synth.random_case(840 + i, N, K, ldq=(N + 15) // 16 * 16)
        weights.append((Q, s, N, K))
    _fused_steps(weights, steps=4, with_bits=with_bits, seed=2 + with_bits)


@pytest.mark.parametrize("with_bits", [True, False])
def test_group_decode_lif_two_launch_form(with_bits):
    """A K above the fused form's 6144 columns takes the two-launch route
    (producer into the spike words or the group's staging, then the decode):
    the same results."""
    shapes = [(304, 8192), (1536, 1536), (48, 7000)]
    weights = []
    for i, (N, K) in enumerate(shapes):
        Q, s, _ = synth.random_case(850 + i, N, K, ldq=(N + 15) // 16 * 16)
        weights.append((Q, s, N, K))
    _fused_steps(weights, steps=3, with_bits=with_bits, seed=4 + with_bits)


def test_group_decode_lif_rejects_overlap_and_alignment():
    weights = synth.decode_step_weights(0, blocks=1)
    plans = [sp.Plan(to_dev(Q), to_dev(s), N, K) for (Q, s, N, K) in weights]
    group = sp.Group(plans)
    n, ld = len(weights), 6144
    a = torch.zeros((n, ld), dtype=torch.float32, device=DEV)
    b = torch.zeros((n, ld), dtype=torch.float32, device=DEV)
    I = torch.zeros((n, ld), dtype=torch.float32, device=DEV)
    bits = torch.zeros((n, ld // 32), dtype=torch.int32, device=DEV)
    y = torch.zeros((n, 1536), dtype=torch.float32, device=DEV)
    lib = sp.lib()
    h, s = group.handle, None

    def call(vin, vout, cur, bt, ldb=ld // 32, ld_=ld):
        return lib.spike_proj_group_decode_lif(h, vin, vout, cur, ld_, 0.9, 1.0, bt, ldb, None,
                                               y.data_ptr(), 1536, s)

    assert call(a.data_ptr(), a.data_ptr(), I.data_ptr(), None) == sp.SP_EINVAL       # in place
    assert call(a.data_ptr(), b.data_ptr() - 64, b.data_ptr(), None) == sp.SP_EINVAL  # v_out over I
    assert call(a.data_ptr(), b.data_ptr(), I.data_ptr(), a.data_ptr() + 4096) == sp.SP_EINVAL
    assert call(a.data_ptr(), b.data_ptr(), I.data_ptr(), bits.data_ptr(), ldb=191) == sp.SP_EINVAL
    assert call(a.data_ptr(), b.data_ptr(), I.data_ptr(), None, ld_=6143) == sp.SP_EINVAL
    assert call(a.data_ptr() + 2, b.data_ptr(), I.data_ptr(), None) == sp.SP_EALIGN
    assert call(a.data_ptr(), b.data_ptr(), I.data_ptr(), bits.data_ptr()) == sp.SP_OK
    torch.cuda.synchronize()
    assert group.status() == sp.SP_OK
