"""Seeded synthetic inputs for the spike-gated INT8 projection.

This module only *makes inputs*: spike masks, INT8 weights and FP32 scales
with the shapes and distributions of the workloads below.  It contains none
of the projection's arithmetic; the CUDA library and the CPU oracle both
consume what it returns and each computes the projection on its own.

The paper's real spikes come from an unreleased checkpoint (Section 6,
Artifact Availability) and it never reports a firing rate, so seeded
Bernoulli spikes stand in for them.  Shapes follow Section 2.1 (22 blocks,
d = 1536) and Appendix A.2 (the feed-forward down projection is 1536 outputs
by 6144 inputs: its INT4 group-scale shape [1536, 192] at group size 32).

Layouts produced here:

* weights ``Q``: INT8, column-major over the logical [N out, K in] matrix
  (Section 2.2), held as a numpy array of shape [K, ldq] whose row k is the
  contiguous column k, so element (m, k) sits at flat offset ``k*ldq + m``.
* scales ``s``: float32 [N], one per output channel (Section 2.3).
* spikes: ``u8`` rows of K bytes in {0, 1}, or ``bits`` rows of
  ceil(K/32) uint32 words, column k at bit k%32 of word k//32, tail bits 0.

All randomness is numpy PCG64 seeded from ``(workload id, seed, index...)``.
"""
from __future__ import annotations

import numpy as np

D_MODEL = 1536            # residual width, Section 2.1
D_FFN = 4 * D_MODEL       # 6144: down-projection input width, Appendix A.2
N_BLOCKS = 22             # decoder blocks, Section 2.1

# workload ids used as the first word of every seed sequence
_W_SINGLE, _W_DOWN, _W_STEP, _W_BATCH, _W_PREFILL, _W_DENSE, _W_MISC = 1, 2, 3, 4, 5, 6, 9
_W_HEAD = 10
VOCAB = 57344             # output vocabulary slots of the deployed configuration (Section 2.1)


def rng_for(*words: int) -> np.random.Generator:
    """PCG64 generator for a tuple of non-negative integer seed words."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(
        [int(w) for w in words])))


# --------------------------------------------------------------------------
# formats
# --------------------------------------------------------------------------
def pack_bits(x_u8: np.ndarray) -> np.ndarray:
    """u8 spikes [..., K] -> uint32 words [..., ceil(K/32)], LSB first.

    Pure format conversion: bit k%32 of word k//32 is (x[k] != 0); bits past
    K are zero."""
    x = np.asarray(x_u8) != 0
    K = x.shape[-1]
    words = (K + 31) // 32
    pad = words * 32 - K
    if pad:
        x = np.concatenate([x, np.zeros(x.shape[:-1] + (pad,), bool)], -1)
    by = np.packbits(x, axis=-1, bitorder="little")
    return np.ascontiguousarray(by).view("<u4").astype(np.uint32)


def unpack_bits(bits: np.ndarray, K: int) -> np.ndarray:
    """uint32 words [..., W] -> u8 spikes [..., K] in {0, 1}."""
    by = np.ascontiguousarray(np.asarray(bits, dtype="<u4")).view(np.uint8)
    return np.unpackbits(by, axis=-1, bitorder="little")[..., :K].astype(np.uint8)


def bernoulli(rng: np.random.Generator, shape, p) -> np.ndarray:
    """u8 spikes: 1 where U(0,1) < p (p broadcast against ``shape``)."""
    return (rng.random(shape) < p).astype(np.uint8)


# --------------------------------------------------------------------------
# weights
# --------------------------------------------------------------------------
def quantise_per_channel(W: np.ndarray):
    """Per-output-channel symmetric INT8 export of a float matrix
    W [N out, K in] (Section 2.3):

        s_m = max(max_k |W_mk|, 1e-8) / 127,  Q_mk = clip(round(W_mk / s_m), -127, 127)

    in float32 with round-half-to-even.  This is the paper's offline export
    step that *produces* the stored weights; it is not part of the
    projection, and both the library and the oracle take its output as
    given.  Returns (Q column-major [K, N] int8, s [N] float32)."""
    W = np.asarray(W, dtype=np.float32)
    amax = np.max(np.abs(W), axis=1)
    s = (np.maximum(amax, np.float32(1e-8)) / np.float32(127.0)).astype(np.float32)
    q = np.clip(np.rint(W / s[:, None]), -127, 127).astype(np.int8)
    return np.ascontiguousarray(q.T), s


def quantised_normal(rng: np.random.Generator, N: int, K: int):
    """W ~ N(0, 1) [N, K] float32, exported per channel: (Q [K, N], s [N])."""
    W = rng.standard_normal((N, K), dtype=np.float32)
    return quantise_per_channel(W)


def uniform_int8(rng: np.random.Generator, N: int, K: int):
    """Q uniform on the integers [-127, 127] with scale
    s_m = max_k |Q_mk| * U(0.5, 1.5) / 127 (float64, stored float32).
    Returns (Q column-major [K, N], s [N])."""
    Qc = rng.integers(-127, 128, size=(K, N), dtype=np.int16).astype(np.int8)
    amax = np.abs(Qc.astype(np.int32)).max(axis=0).astype(np.float64)
    u = rng.uniform(0.5, 1.5, size=N)
    s = (amax * u / 127.0).astype(np.float32)
    return np.ascontiguousarray(Qc), s


# --------------------------------------------------------------------------
# workloads
# --------------------------------------------------------------------------
def single_projection(seed: int = 0, N: int = D_MODEL, K: int = D_MODEL,
                      p: float = 0.1):
    """Single spike projection, batch 1: K = N = 1536, x ~ Bernoulli(0.1),
    uniform INT8 W, scale max|w_row| * U(0.5, 1.5) / 127."""
    rng = rng_for(_W_SINGLE, seed)
    Q, s = uniform_int8(rng, N, K)
    x = bernoulli(rng, (K,), p)
    return dict(Q=Q, s=s, N=N, K=K, x=x, bits=pack_bits(x))


def down_weights(seed: int = 0, N: int = D_MODEL, K: int = D_FFN):
    """FFN down projection weights: K = 6144 in, N = 1536 out, N(0,1)
    quantised per output channel."""
    return quantised_normal(rng_for(_W_DOWN, seed), N, K)


DOWN_RATES = (0.02, 0.05, 0.1, 0.2, 0.5)


def down_spikes(p: float, count: int = 1000, seed: int = 0, K: int = D_FFN):
    """``count`` i.i.d. Bernoulli(p) spike vectors for the down projection
    (u8 [count, K])."""
    rng = rng_for(_W_DOWN, seed, int(round(p * 1e6)))
    return bernoulli(rng, (count, K), p)


def decode_step_weights(seed: int = 0, blocks: int = N_BLOCKS):
    """Weights of a 22-block decode step: per block a TCAM projection
    (1536 -> 1536) and a down projection (6144 -> 1536), each seeded on its
    own.  Returns a list of 2*blocks (Q, s, N, K) tuples in the order
    [tcam_0, down_0, tcam_1, down_1, ...]."""
    out = []
    for b in range(blocks):
        for j, K in enumerate((D_MODEL, D_FFN)):
            Q, s = quantised_normal(rng_for(_W_STEP, seed, b, j), D_MODEL, K)
            out.append((Q, s, D_MODEL, K))
    return out


def decode_step_spikes(step: int, Ks, p: float = 0.1, seed: int = 0):
    """Fresh Bernoulli(p) spikes for every projection of one decode step:
    list of u8 vectors, one per entry of ``Ks``."""
    out = []
    for j, K in enumerate(Ks):
        rng = rng_for(_W_STEP, seed, 1_000_000 + step, j)
        out.append(bernoulli(rng, (K,), p))
    return out


def batched_spikes(seed: int = 0, B: int = 64, K: int = D_FFN,
                   correlated: bool = False, hot_frac: float = 0.1,
                   hot_share: float = 0.7):
    """Batched decode spikes u8 [B, K]; token rates p_t ~ U(0.05, 0.2).

    Independent: x[t, k] ~ Bernoulli(p_t).  Correlated: a hot set H of
    round(hot_frac*K) columns shared by all tokens supplies ``hot_share`` of
    each token's expected actives: hot columns fire with
    q_h = min(1, hot_share*p_t*K/|H|), the others with the rate that keeps
    the token's expected count at p_t*K.  Where q_h clamps at 1 the realised
    hot share falls below ``hot_share``.  Returns (x, p_t, H)."""
    rng = rng_for(_W_BATCH, seed, int(correlated))
    p_t = rng.uniform(0.05, 0.2, size=B)
    if not correlated:
        return bernoulli(rng, (B, K), p_t[:, None]), p_t, np.zeros(0, np.int64)
    nh = int(round(hot_frac * K))
    H = np.sort(rng.choice(K, size=nh, replace=False))
    q_h = np.minimum(1.0, hot_share * p_t * K / nh)
    q_c = np.clip((p_t * K - nh * q_h) / (K - nh), 0.0, 1.0)
    is_hot = np.zeros(K, bool)
    is_hot[H] = True
    rate = np.where(is_hot[None, :], q_h[:, None], q_c[:, None])
    return bernoulli(rng, (B, K), rate), p_t, H


def prefill_spikes(block: int = 0, seed: int = 0, T: int = 512,
                   K: int = D_FFN, p: float = 0.15, sigma: float = 0.5):
    """512-token prefill spikes u8 [T, K]: column rates
    p_k = min(1, p * exp(sigma * z_k)), z ~ N(0, 1) (log-normal(0, sigma)
    multipliers), then X[t, k] ~ Bernoulli(p_k)."""
    rng = rng_for(_W_PREFILL, seed, block)
    rate = np.minimum(1.0, p * np.exp(sigma * rng.standard_normal(K)))
    return bernoulli(rng, (T, K), rate[None, :])


def prefill_weights(block: int = 0, seed: int = 0):
    """Down-projection weights of one prefill block (N(0,1) exported)."""
    return quantised_normal(rng_for(_W_PREFILL, seed, 1000 + block),
                            D_MODEL, D_FFN)


def random_case(seed: int, N: int, K: int, T: int = 1, p: float = 0.1,
                ldq: int | None = None, weights: str = "uniform"):
    """Small generic case for parity tests: Q [K, ldq] (column-major with
    leading dimension ldq >= N, padding bytes random), s [N], x u8 [T, K]."""
    rng = rng_for(_W_MISC, seed, N, K, T)
    ldq = N if ldq is None else ldq
    if weights == "uniform":
        Q = rng.integers(-128, 128, size=(K, ldq), dtype=np.int16).astype(np.int8)
    elif weights == "normal":
        Qn, _ = quantised_normal(rng, ldq, K)
        Q = Qn
    else:
        raise ValueError(weights)
    s = rng.uniform(-2.0, 2.0, size=N).astype(np.float32)
    x = bernoulli(rng, (T, K), p)
    return np.ascontiguousarray(Q), s, x


# --------------------------------------------------------------------------
# continuous-input projections (row-major INT8 weights, FP32 activations)
# --------------------------------------------------------------------------
# Per block, the projections that read the continuous stream (Section 2.1):
# fused query/key/value (3 x 1536 out), attention output (1536 out) and FFN up
# (6144 out), all with 1536 inputs.  The paper does not give their exact
# shapes; these follow the stated residual width and FFN width.
DENSE_KINDS = {"qkv": 3 * D_MODEL, "out": D_MODEL, "up": D_FFN}


def dense_weights(block: int, kind: str, seed: int = 0, K: int = D_MODEL):
    """Row-major INT8 weights [N, K] and scale [N] of one continuous-input
    projection of block ``block``: N(0, 1) exported per output channel
    (the same export as the spike-gated weights, transposed to row-major)."""
    N = DENSE_KINDS[kind]
    Qc, s = quantised_normal(rng_for(_W_DENSE, seed, block, list(DENSE_KINDS).index(kind)), N, K)
    return np.ascontiguousarray(Qc.T), s


def hidden_state(step: int, B: int = 1, seed: int = 0, K: int = D_MODEL):
    """Continuous activations x ~ N(0, 1), float32 [B, K]."""
    return rng_for(_W_DENSE, seed, 10_000 + step).standard_normal((B, K), dtype=np.float32)


# --------------------------------------------------------------------------
# vocabulary head (Section 5, trace configuration)
# --------------------------------------------------------------------------
HEAD_LOGIT_STD = 2.5


def head_weights(seed: int = 0, V: int = VOCAB, K: int = D_MODEL,
                 logit_std: float = HEAD_LOGIT_STD):
    """Row-major INT8 head weights [V, K] and scale [V]: W ~ N(0, sigma^2)
    with sigma = logit_std / sqrt(K), exported per output row (Section 2.3).
    With N(0, 1) hidden states the logits then have standard deviation near
    logit_std, and the top-two gap of 57,344 of them falls below 0.5 in
    roughly the share of steps the paper's trace reports (54 of 80)."""
    rng = rng_for(_W_HEAD, seed, V, K)
    sigma = np.float32(logit_std / np.sqrt(K))
    Qc = np.empty((K, V), dtype=np.int8)
    s = np.empty(V, dtype=np.float32)
    step = 8192
    for m0 in range(0, V, step):            # row blocks: bounded float32 scratch
        W = rng.standard_normal((min(step, V - m0), K), dtype=np.float32) * sigma
        q, sb = quantise_per_channel(W)
        Qc[:, m0:m0 + W.shape[0]] = q
        s[m0:m0 + W.shape[0]] = sb
    return np.ascontiguousarray(Qc.T), s


def head_hidden(step: int, B: int = 1, seed: int = 0, K: int = D_MODEL):
    """Final hidden states h ~ N(0, 1), float32 [B, K] (post-normalisation
    scale)."""
    return rng_for(_W_HEAD, seed, 20_000 + step).standard_normal((B, K), dtype=np.float32)

