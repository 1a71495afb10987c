"""Vocabulary head (spike_proj_head) against the CPU oracle (GPU): the
approximate logits, the top-two gap, the gate decision and the candidate
rows bit for bit; the recomputed logits within the FP32 dot-product bound;
the token equal to the oracle's wherever the exact logits decide it, and
otherwise a candidate whose exact logit is within the bound of the best.
Covers ragged V and K (unit and chunk tails), 1-4 hidden states, k_sel 1-64,
tau 0 / 0.5 / 4 / inf, ties, the smallest vocabularies, repeated calls (the
tickets reset), the full 57,344 x 1536 head, and argument errors."""
import ctypes
import functools
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu

U = 2.0 ** -24


def r_bound(K, s, mag, r_ref):
    """|r - r_exact| allowed: gamma(d) |s| sum|W h| + 2u |r| (depth d of the
    per-lane chains plus the butterfly)."""
    d = 16 * math.ceil(K / 512) + 5
    g = d * U / (1 - d * U)
    return np.abs(s) * g * mag + 2 * U * np.abs(r_ref) + 1e-45


def small_case(seed, V, K, ldw=None, logit_std=2.5):
    rng = synth.rng_for(7800, seed, V, K)
    ldw = (K + 15) // 16 * 16 if ldw is None else ldw
    W = rng.standard_normal((V, K)).astype(np.float32) * np.float32(logit_std / math.sqrt(K))
    Qc, s = synth.quantise_per_channel(W)
    Q = np.zeros((V, ldw), np.int8)
    Q[:, :K] = Qc.T
    Q[:, K:] = rng.integers(-127, 128, size=(V, ldw - K))       # padding: never used
    return Q, s


@functools.lru_cache(maxsize=1)
def full_head():
    Q, s = synth.head_weights()
    return Q, s, to_dev(Q), to_dev(s)


def run_head(head, h, tau, k_sel, V):
    B = h.shape[0]
    hd = to_dev(h)
    token = torch.full((B,), -7, dtype=torch.int32, device=DEV)
    verified = torch.full((B,), -7, dtype=torch.int32, device=DEV)
    gap = torch.full((B,), float("nan"), dtype=torch.float32, device=DEV)
    cand = torch.full((B, k_sel), -7, dtype=torch.int32, device=DEV)
    r = torch.full((B, k_sel), float("nan"), dtype=torch.float32, device=DEV)
    z = torch.full((B, V + 3), float("nan"), dtype=torch.float32, device=DEV)
    head(hd, tau, k_sel, token, verified, gap, cand, r, z)
    torch.cuda.synchronize()
    return {"token": token.cpu().numpy(), "verified": verified.cpu().numpy(),
            "gap": gap.cpu().numpy(), "cand": cand.cpu().numpy(), "r": r.cpu().numpy(),
            "z": z.cpu().numpy()}


def check(got, Q, s, V, K, h, tau, k_sel, what):
    want = oracle.head(Q, s, V, K, h, tau, k_sel, ldq=Q.shape[1])
    B = h.shape[0]
    assert np.array_equal(got["z"][:, :V].view(np.uint32), want["z"].view(np.uint32)), \
        f"{what}: approximate logits differ"
    assert np.all(np.isnan(got["z"][:, V:])), f"{what}: wrote past V"
    assert np.array_equal(got["gap"], want["gap"]), f"{what}: gap"
    assert np.array_equal(got["verified"], want["verified"]), f"{what}: gate"
    assert np.array_equal(got["cand"], want["cand"]), f"{what}: candidates"
    for b in range(B):
        c = want["cand"][b]
        if not want["verified"][b]:
            assert got["token"][b] == c[0], f"{what}: token without verification"
            assert np.all(np.isnan(got["r"][b])), f"{what}: r written without verification"
            continue
        rg = got["r"][b].astype(np.float64)
        bound = r_bound(K, s[c].astype(np.float64), want["r_abs"][b], want["r"][b])
        assert np.all(np.abs(rg - want["r"][b]) <= bound), f"{what}: recomputed logits"
        # the GPU's decision on its own values: largest r, equal r lower row
        order = sorted(range(k_sel), key=lambda i: (-rg[i], c[i]))
        assert got["token"][b] == c[order[0]], f"{what}: token is not the argmax of r"
        # against the exact logits: unique when the best clears every other
        # candidate by both bounds, else any candidate within them is valid
        ex, tb = want["r"][b], int(want["token"][b])
        ib = int(np.where(c == tb)[0][0])
        ig = int(np.where(c == got["token"][b])[0][0])
        assert ex[ig] + bound[ig] >= ex[ib] - bound[ib], f"{what}: token not within bound"
        if np.all((ex[ib] - bound[ib] > ex + bound) | (np.arange(k_sel) == ib)):
            assert got["token"][b] == tb, f"{what}: token differs where the exact logits decide"


@pytest.mark.parametrize("V,K", [(5001, 1000), (4096, 1536), (999, 40), (70, 512), (2, 16),
                                 (1500, 2048), (1200, 2049), (1000, 8192)])
@pytest.mark.parametrize("B", [1, 2, 4])
def test_head_vs_oracle(V, K, B):
    Q, s = small_case(1, V, K)
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    # row pitch a multiple of 4 floats past K (the API's rule for h)
    h = synth.rng_for(7801, V, K, B).standard_normal((B, (K + 3) // 4 * 4 + 4)).astype(np.float32)
    for tau in (0.0, 0.5, np.inf):
        for k_sel in sorted({1, min(16, V), min(64, V)}):
            got = run_head(head, h, tau, k_sel, V)
            check(got, Q, s, V, K, h, tau, k_sel, f"V={V} K={K} B={B} tau={tau} k={k_sel}")


def test_head_b3_and_padded_rows():
    V, K = 3000, 777
    Q, s = small_case(2, V, K, ldw=800)
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    h = synth.rng_for(7802).standard_normal((3, 780)).astype(np.float32)
    check(run_head(head, h, np.inf, 64, V), Q, s, V, K, h, np.inf, 64, "B=3 padded")


def test_head_ties():
    """Duplicate rows give equal logits: candidates by ascending row, the
    verified token the lower row of a tied best."""
    V, K = 2000, 256
    Q, s = small_case(3, V, K)
    h = synth.rng_for(7803).standard_normal((1, K)).astype(np.float32)
    want = oracle.head(Q, s, V, K, h, np.inf, 8, ldq=Q.shape[1])
    best = int(want["cand"][0][0])
    dsts = [d for d in (1999, 3, 1000) if d != best]
    for dst in dsts:
        Q[dst], s[dst] = Q[best], s[best]
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    got = run_head(head, h, np.inf, 8, V)
    check(got, Q, s, V, K, h, np.inf, 8, "ties")
    assert got["gap"][0] == 0.0 and got["verified"][0] == 1
    assert got["token"][0] == min([best] + dsts)


def test_head_gate_boundary():
    """tau equal to the gap does not verify (strict), the next float does."""
    V, K = 1500, 300
    Q, s = small_case(4, V, K)
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    h = synth.rng_for(7804).standard_normal((1, K)).astype(np.float32)
    g = run_head(head, h, 0.0, 4, V)["gap"][0]
    assert run_head(head, h, float(g), 4, V)["verified"][0] == 0
    up = float(np.nextafter(np.float32(g), np.float32(np.inf)))
    got = run_head(head, h, up, 4, V)
    assert got["verified"][0] == 1
    check(got, Q, s, V, K, h, up, 4, "gate boundary")


def test_head_repeated_calls():
    """Many calls in a row, the tickets reset by each: every result right."""
    V, K = 20000, 1536
    Q, s = small_case(5, V, K)
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    for step in range(12):
        h = synth.head_hidden(step, B=1 + step % 4)
        check(run_head(head, h, 0.5, 32, V), Q, s, V, K, h, 0.5, 32, f"step {step}")


@pytest.mark.parametrize("k_sel", [16, 32, 64])
def test_head_full_size(k_sel):
    """The deployed head, 57,344 x 1536, at the trace gate (0.5) and the
    power gate (4.0), four hidden states per call."""
    Q, s, Qd, sd = full_head()
    V, K = Q.shape
    head = sp.Head(Qd, sd, K=K)
    for step, tau in ((0, 0.5), (1, 4.0)):
        h = synth.head_hidden(100 + step, B=4)
        check(run_head(head, h, tau, k_sel, V), Q, s, V, K, h, tau, k_sel,
              f"full k={k_sel} tau={tau}")


def test_head_outputs_optional():
    V, K = 1000, 128
    Q, s = small_case(6, V, K)
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    h = synth.rng_for(7806).standard_normal((2, K)).astype(np.float32)
    token = torch.zeros(2, dtype=torch.int32, device=DEV)
    head(to_dev(h), np.inf, 16, token)
    torch.cuda.synchronize()
    want = run_head(head, h, np.inf, 16, V)
    assert np.array_equal(token.cpu().numpy(), want["token"])


def test_head_errors():
    V, K = 256, 64
    Q, s = small_case(7, V, K)
    Qd, sd = to_dev(Q), to_dev(s)
    lib = sp.lib()
    h = ctypes.c_void_p()
    assert lib.spike_proj_head_create(ctypes.byref(h), Qd.data_ptr(), 64, sd.data_ptr(), 1, K,
                                      None) == sp.SP_ERANGE          # V < 2
    assert lib.spike_proj_head_create(ctypes.byref(h), Qd.data_ptr(), 64, sd.data_ptr(), V, 8193,
                                      None) == sp.SP_ERANGE          # K above the cap
    assert lib.spike_proj_head_create(ctypes.byref(h), Qd.data_ptr(), 72, sd.data_ptr(), V, K,
                                      None) == sp.SP_EALIGN          # ldw % 16
    assert lib.spike_proj_head_create(ctypes.byref(h), Qd.data_ptr() + 8, 64, sd.data_ptr(), V, K,
                                      None) == sp.SP_EALIGN          # W alignment
    head = sp.Head(Qd, sd, K=K)
    hd = torch.zeros((4, 64), dtype=torch.float32, device=DEV)
    tok = torch.zeros(4, dtype=torch.int32, device=DEV)
    hh = head.handle

    def call(hp, ldh, B, k, tk=tok.data_ptr(), z=None, ldz=0):
        return lib.spike_proj_head(hh, hp, ldh, B, 0.5, k, tk, None, None, None, None, z, ldz, None)

    assert call(hd.data_ptr(), 64, 0, 16) == sp.SP_EINVAL              # B
    assert call(hd.data_ptr(), 64, 5, 16) == sp.SP_EINVAL
    assert call(hd.data_ptr(), 64, 1, 0) == sp.SP_EINVAL               # k_sel
    assert call(hd.data_ptr(), 64, 1, 65) == sp.SP_EINVAL
    assert call(hd.data_ptr(), 60, 1, 16) == sp.SP_EINVAL              # ldh < K
    assert call(hd.data_ptr(), 68, 1, 16) == sp.SP_OK
    assert call(hd.data_ptr() + 4, 64, 1, 16) == sp.SP_EALIGN          # h alignment
    assert call(hd.data_ptr(), 66, 1, 16) == sp.SP_EALIGN              # ldh % 4
    assert call(hd.data_ptr(), 64, 1, 16, z=hd.data_ptr(), ldz=100) == sp.SP_EINVAL   # ld_z < V
    assert call(hd.data_ptr(), 64, 1, 16, tk=0) == sp.SP_EINVAL        # token required
    torch.cuda.synchronize()
    small = sp.Head(Qd[:5], sd[:5], K=K)
    assert lib.spike_proj_head(small.handle, hd.data_ptr(), 64, 1, 0.5, 6, tok.data_ptr(), None,
                               None, None, None, None, 0, None) == sp.SP_EINVAL   # k_sel > V


@pytest.mark.parametrize("V,K", [(3000, 256), (57344, 1536)])
def test_head_equal_logits(V, K):
    """A zero hidden state makes every approximate logit 0: the histogram
    bound passes every listed key, so the selection merges every list (the
    exact slow path). Candidates are then the lowest rows, the gap is 0 and
    the recomputed logits are all 0."""
    if V == 57344:
        Q, s, Qd, sd = full_head()
    else:
        Q, s = small_case(8, V, K)
        Qd, sd = to_dev(Q), to_dev(s)
    head = sp.Head(Qd, sd, K=K)
    h = np.zeros((2, K), np.float32)
    got = run_head(head, h, 0.5, 64, V)
    check(got, Q, s, V, K, h, 0.5, 64, f"equal logits V={V}")
    assert np.array_equal(got["cand"][0], np.arange(64))
    assert got["token"][0] == 0 and got["gap"][0] == 0.0
    # and the call after it is fast-path again and right
    h2 = synth.head_hidden(7, B=2, K=K)
    check(run_head(head, h2, 0.5, 64, V), Q, s, V, K, h2, 0.5, 64, "after equal logits")


def test_head_codes_at_exact_halves():
    """Hidden values whose quotient by s_x is exactly an integer plus one half
    (s_x a power of two): the codes round half to even as IEEE division
    does, so the approximate logits match the oracle bit for bit."""
    V, K = 512, 1024
    Q, s = small_case(9, V, K)
    rng = synth.rng_for(7809)
    q = rng.integers(-126, 127, size=(2, K)).astype(np.float64) + 0.5
    q[:, 0] = 127.0
    q[1, 0] = -127.0
    q[:, 1::7] = np.round(q[:, 1::7])                # some exact integers too
    h = (q * 2.0 ** -5).astype(np.float32)          # s_x = 127 * 2^-5 / 127 = 2^-5 exactly
    head = sp.Head(to_dev(Q), to_dev(s), K=K)
    got = run_head(head, h, np.inf, 16, V)
    check(got, Q, s, V, K, h, np.inf, 16, "exact halves")
