"""Seeded input generators: formats, the export step, distributions (no GPU)."""
import numpy as np

from paper_2606_03026_gb300 import synth


def test_pack_unpack_roundtrip():
    rng = synth.rng_for(1)
    for K in (1, 31, 32, 33, 100, 6144):
        x = synth.bernoulli(rng, (3, K), 0.4)
        b = synth.pack_bits(x)
        assert b.dtype == np.uint32 and b.shape == (3, (K + 31) // 32)
        assert np.array_equal(synth.unpack_bits(b, K), x)
        # LSB-first: column k is bit k%32 of word k//32; tail bits are zero
        for k in range(K):
            assert ((b[0, k // 32] >> (k % 32)) & 1) == x[0, k]
        if K % 32:
            assert (b[:, -1] >> np.uint32(K % 32) == 0).all()


def test_quantiser_matches_section_2_3():
    rng = synth.rng_for(2)
    W = rng.standard_normal((64, 300)).astype(np.float32)
    W[5] = 0.0                                   # all-zero row: floor 1e-8
    Qc, s = synth.quantise_per_channel(W)
    Q = Qc.T.astype(np.int32)
    assert Qc.shape == (300, 64) and s.shape == (64,)
    assert np.all(np.abs(Q) <= 127)
    amax = np.abs(W).max(axis=1)
    ok = amax > 0
    assert np.allclose(s[ok] * 127, amax[ok], rtol=1e-6)
    assert s[5] == np.float32(np.float32(1e-8) / np.float32(127)) and not Q[5].any()
    # round to nearest: |W/s - Q| <= 1/2 away from the clip
    r = W[ok] / s[ok, None]
    assert np.all(np.abs(r - Q[ok]) <= 0.5 + 1e-5)
    # each row's largest |W| maps to +-127
    am = np.argmax(np.abs(W[ok]), axis=1)
    assert np.all(np.abs(Q[ok][np.arange(ok.sum()), am]) == 127)


def test_uniform_weights_and_scale():
    Q, s = synth.uniform_int8(synth.rng_for(3), 1536, 1536)
    assert Q.shape == (1536, 1536) and Q.min() >= -127 and Q.max() <= 127
    amax = np.abs(Q.astype(np.int32)).max(axis=0)
    ratio = s.astype(np.float64) * 127 / amax
    assert ratio.min() >= 0.5 - 1e-6 and ratio.max() <= 1.5 + 1e-6


def test_workload_shapes_and_rates():
    c1 = synth.single_projection(0)
    assert c1["x"].shape == (1536,) and abs(c1["x"].mean() - 0.1) < 0.03
    x = synth.down_spikes(0.05, count=200)
    assert x.shape == (200, 6144) and abs(x.mean() - 0.05) < 0.005
    xb, p_t, _ = synth.batched_spikes(0, correlated=False)
    assert xb.shape == (64, 6144) and np.all((p_t >= 0.05) & (p_t <= 0.2))
    assert abs(xb.mean(axis=1) - p_t).max() < 0.02
    xc, p_c, H = synth.batched_spikes(0, correlated=True)
    assert len(H) == 614
    hot_share = xc[:, H].sum() / xc.sum()
    assert 0.55 < hot_share < 0.72      # 0.7 target, lower where q_h clamps
    X = synth.prefill_spikes(0)
    assert X.shape == (512, 6144) and 0.15 < X.mean() < 0.19


def test_seeded_reproducible():
    a = synth.single_projection(0)
    b = synth.single_projection(0)
    c = synth.single_projection(1)
    assert np.array_equal(a["Q"], b["Q"]) and np.array_equal(a["x"], b["x"])
    assert not np.array_equal(a["x"], c["x"])


def test_head_inputs():
    """The vocabulary head's stand-in weights: row-major [V, K] INT8 with the
    Section 2.3 export (every row reaches +-127 at its largest magnitude),
    logits of about the stated spread, seeded and reproducible."""
    Q, s = synth.head_weights(V=4096, K=1536)
    assert Q.shape == (4096, 1536) and Q.dtype == np.int8 and s.shape == (4096,)
    assert np.all(np.abs(Q.astype(np.int16)).max(axis=1) == 127)
    Q2, s2 = synth.head_weights(V=4096, K=1536)
    assert np.array_equal(Q, Q2) and np.array_equal(s, s2)
    h = synth.head_hidden(0, B=64)
    z = (Q.astype(np.float64) * s[:, None]) @ h.T.astype(np.float64)
    assert abs(z.std() - synth.HEAD_LOGIT_STD) < 0.2 * synth.HEAD_LOGIT_STD
    assert not np.array_equal(synth.head_hidden(0), synth.head_hidden(1))


def test_dense_inputs():
    """Continuous-input stand-ins: row-major weights of the stated shapes with
    the per-row export, and N(0, 1) hidden states."""
    for kind, N in synth.DENSE_KINDS.items():
        W, s = synth.dense_weights(0, kind)
        assert W.shape == (N, synth.D_MODEL) and W.dtype == np.int8 and s.shape == (N,)
        assert np.all(np.abs(W.astype(np.int16)).max(axis=1) == 127)
    x = synth.hidden_state(0, B=4)
    assert x.shape == (4, synth.D_MODEL) and x.dtype == np.float32
    assert abs(float(x.std()) - 1.0) < 0.05
