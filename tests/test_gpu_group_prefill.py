"""Grouped prefill: the dense tensor-core contraction (ACC = X Q^T, Y = ACC * s
per column; Eq. (sparse) for every row, the 512-token prefill of Section 3.2)
for every member of a group in one persistent launch, through the C ABI,
against the CPU oracle (GPU)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import DEV, assert_parity, to_dev
from paper_2606_03026_gb300 import spikeproj as sp
from paper_2606_03026_gb300 import synth

pytestmark = pytest.mark.gpu

# ragged members: N not a multiple of the 256-channel tile, K not a multiple
# of the 64-column K block, padded leading dimensions, one-tile members
RAGGED = [(272, 1000, 288), (48, 64, 48), (1536, 777, 1536), (256, 6143, 256),
          (16, 1, 16), (528, 130, 544)]


def make_members(shapes, T, seed=0, p=0.15):
    members = []
    for i, (N, K, ldq) in enumerate(shapes):
        Q, s, x = synth.random_case(700 + seed * 31 + i, N, K, T=T, p=p, ldq=ldq)
        plan = sp.Plan(to_dev(Q), to_dev(s), N, K, ldw=ldq, max_batch=max(T, 1), gemm=True)
        members.append((Q, s, x, N, K, ldq, plan))
    return members


def run_group(group, members, xs_dev, fmt, T, ldx, with_acc=True, with_y=True):
    accs = [torch.full((T, m[3]), -7, dtype=torch.int32, device=DEV) for m in members]
    ys = [torch.full((T, m[3]), -7.0, dtype=torch.float32, device=DEV) for m in members]
    group.prefill(xs_dev, fmt, T, ldx, accs if with_acc else None, ys if with_y else None)
    torch.cuda.synchronize()
    return accs, ys


@pytest.mark.parametrize("T", [1, 129, 200])
@pytest.mark.parametrize("fmt", ["bool8", "u8", "bits"])
def test_ragged_group(T, fmt):
    """Members of different N, K and ldw in one launch, every output against
    the oracle; bool8 rows are read in place, u8 and bit rows staged."""
    members = make_members(RAGGED, T, seed=T)
    group = sp.Group([m[-1] for m in members])
    Kmax = max(m[4] for m in members)
    if fmt == "bits":
        ldx = (Kmax + 31) // 32
        rows = [np.zeros((T, ldx), np.uint32) for _ in members]
        for r, m in zip(rows, members):
            b = synth.pack_bits(m[2])
            r[:, : b.shape[1]] = b
    else:
        ldx = (Kmax + 15) // 16 * 16
        rows = [np.zeros((T, ldx), np.uint8) for _ in members]
        for r, m in zip(rows, members):
            r[:, : m[4]] = m[2] if fmt == "bool8" else m[2] * 3   # u8: any nonzero fires
    xs_dev = [to_dev(r) for r in rows]
    accs, ys = run_group(group, members, xs_dev, fmt, T, ldx)
    for j, (Q, s, x, N, K, ldq, _) in enumerate(members):
        want_acc, want_y = oracle.project(Q, s, N, K, x, "u8", ldq=ldq)
        assert_parity(accs[j], ys[j], want_acc, want_y, f"member {j} ({N}x{K}) {fmt} T={T}")
    assert group.status() == sp.SP_OK
    group.close()


def test_outputs_optional_and_unaligned_rows():
    """acc only, y only, and bool8 rows at an odd byte offset (staged, not
    read in place): same results."""
    T = 131
    members = make_members(RAGGED[:4], T, seed=5)
    group = sp.Group([m[-1] for m in members])
    Kmax = max(m[4] for m in members)
    ldx = (Kmax + 15) // 16 * 16 + 16
    buf = [torch.zeros(T * ldx + 1, dtype=torch.uint8, device=DEV) for _ in members]
    xs_dev = []
    for b, m in zip(buf, members):
        view = b[1:].view(T, ldx)
        view[:, : m[4]] = to_dev(m[2])
        xs_dev.append(view)
    wants = [oracle.project(Q, s, N, K, x, "u8", ldq=ldq) for (Q, s, x, N, K, ldq, _) in members]
    accs, _ = run_group(group, members, xs_dev, "bool8", T, ldx, with_y=False)
    _, ys = run_group(group, members, xs_dev, "bool8", T, ldx, with_acc=False)
    for j, (wa, wy) in enumerate(wants):
        assert_parity(accs[j], ys[j], wa, wy, f"member {j} split outputs")
    group.close()


@pytest.fixture(scope="module")
def prefill22():
    """The 512-token prefill of a 22-block decoder: per block the FFN down
    projection (6144 -> 1536), column rates 0.15 * lognormal(0, 0.5)."""
    blocks = []
    for b in range(22):
        Q, s = synth.prefill_weights(b)
        X = synth.prefill_spikes(b)
        plan = sp.Plan(to_dev(Q), to_dev(s), 1536, 6144, max_batch=512, gemm=True)
        blocks.append((Q, s, X, plan))
    group = sp.Group([b[3] for b in blocks])
    yield blocks, group
    group.close()


def test_prefill_22_blocks(prefill22):
    """22 x (512 x 6144 -> 1536) in one launch, bool8 rows in place: two
    blocks in full and 12 sampled rows of every block against the oracle, and
    every block bit for bit against its own per-plan tensor-core call."""
    blocks, group = prefill22
    T, N, K = 512, 1536, 6144
    xs_dev = [to_dev(X).bool() for (_, _, X, _) in blocks]
    accs = [torch.full((T, N), -7, dtype=torch.int32, device=DEV) for _ in blocks]
    ys = [torch.full((T, N), -7.0, dtype=torch.float32, device=DEV) for _ in blocks]
    group.prefill(xs_dev, "bool8", T, K, accs, ys)
    torch.cuda.synchronize()
    rows = np.array([0, 1, 63, 127, 128, 200, 255, 256, 383, 384, 510, 511])
    for j, (Q, s, X, plan) in enumerate(blocks):
        if j in (0, 21):
            want_acc, want_y = oracle.project(Q, s, N, K, X, "u8")
            assert_parity(accs[j], ys[j], want_acc, want_y, f"block {j} full")
        else:
            want_acc, want_y = oracle.project(Q, s, N, K, X[rows], "u8")
            assert_parity(accs[j][rows], ys[j][rows], want_acc, want_y, f"block {j} rows")
        a1 = torch.empty(T, N, dtype=torch.int32, device=DEV)
        y1 = torch.empty(T, N, dtype=torch.float32, device=DEV)
        plan.batched(xs_dev[j], "bool8", T, K, a1, y1, "gemm")
        torch.cuda.synchronize()
        assert torch.equal(a1, accs[j]), f"block {j}: grouped and per-plan acc differ"
        assert torch.equal(y1.view(torch.int32), ys[j].view(torch.int32)), \
            f"block {j}: grouped and per-plan y differ"
    assert group.status() == sp.SP_OK


def test_prefill_mixed_decoder_group():
    """The 44 binary-input projections of a 22-block decoder (TCAM 1536 ->
    1536 and FFN down 6144 -> 1536 alternating) prefilling 256 tokens in one
    launch: members of different K; sampled rows against the oracle."""
    weights = synth.decode_step_weights(0)
    T = 256
    plans = [sp.Plan(to_dev(Q), to_dev(s), N, K, max_batch=T, gemm=True)
             for (Q, s, N, K) in weights]
    group = sp.Group(plans)
    xs = [synth.prefill_spikes(100 + j, T=T, K=K) for j, (_, _, _, K) in enumerate(weights)]
    ldx = max(w[3] for w in weights)
    rows_np = []
    for x in xs:
        r = np.zeros((T, ldx), np.uint8)
        r[:, : x.shape[1]] = x
        rows_np.append(r)
    xs_dev = [to_dev(r).bool() for r in rows_np]
    accs = [torch.empty(T, w[2], dtype=torch.int32, device=DEV) for w in weights]
    ys = [torch.empty(T, w[2], dtype=torch.float32, device=DEV) for w in weights]
    group.prefill(xs_dev, "bool8", T, ldx, accs, ys)
    torch.cuda.synchronize()
    rows = np.array([0, 5, 127, 128, 255])
    for j, ((Q, s, N, K), x) in enumerate(zip(weights, xs)):
        want_acc, want_y = oracle.project(Q, s, N, K, x[rows], "u8")
        assert_parity(accs[j][rows], ys[j][rows], want_acc, want_y, f"member {j} ({N}x{K})")
    assert group.status() == sp.SP_OK
    group.close()
    for p in plans:
        p.close()


@pytest.mark.parametrize("T,shapes", [
    (256, [(1536, 6144, 1536)] * 3),                  # 2-SM pairs, 18 units split 4 ways
    (100, [(1536, 2000, 1536), (1536, 2048, 1536)]),  # single CTAs, 12 units split 6 ways
    (384, [(1024, 3000, 1024)] * 7 + [(1536, 1536, 1536)] * 9),   # a partial last round
])
def test_tail_split_shapes(T, shapes):
    """Groups whose tiles leave the persistent grid's last round partly idle:
    the tail units run as K ranges on several clusters, the owner adding the
    helpers' fp32 partials.  Every output against the oracle, twice (the
    partials' flags are cleared for the next launch)."""
    members = make_members(shapes, T, seed=len(shapes))
    group = sp.Group([m[-1] for m in members])
    ldx = max(m[4] for m in members)
    xs_dev = []
    for m in members:
        r = np.zeros((T, ldx), np.uint8)
        r[:, : m[4]] = m[2]
        xs_dev.append(to_dev(r).bool())
    wants = [oracle.project(Q, s, N, K, x, "u8", ldq=ldq) for (Q, s, x, N, K, ldq, _) in members]
    for rep in range(2):
        accs, ys = run_group(group, members, xs_dev, "bool8", T, ldx)
        for j, (wa, wy) in enumerate(wants):
            assert_parity(accs[j], ys[j], wa, wy, f"member {j} rep {rep}")
    assert group.status() == sp.SP_OK
    group.close()


def test_group_prefill_errors():
    members = make_members(RAGGED[:2], 8, seed=9)
    plain = sp.Plan(to_dev(members[0][0]), to_dev(members[0][1]), members[0][3], members[0][4],
                    ldw=members[0][5], max_batch=8)
    xs = [to_dev(np.zeros((8, 1024), np.uint8)) for _ in range(2)]
    out = [torch.empty(8, m[3], dtype=torch.int32, device=DEV) for m in members]
    g_plain = sp.Group([plain, members[1][-1]])
    with pytest.raises(sp.SpikeProjError) as e:
        g_plain.prefill(xs, "bool8", 8, 1024, out, None)
    assert e.value.status == sp.SP_EUNSUPPORTED
    g = sp.Group([m[-1] for m in members])
    with pytest.raises(sp.SpikeProjError) as e:          # T above the plans' max_batch
        g.prefill(xs, "bool8", 9, 1024, out, None)
    assert e.value.status == sp.SP_ERANGE
    with pytest.raises(sp.SpikeProjError) as e:          # neither output
        g.prefill(xs, "bool8", 8, 1024, None, None)
    assert e.value.status == sp.SP_EINVAL
    with pytest.raises(sp.SpikeProjError) as e:          # rows shorter than K
        g.prefill(xs, "bool8", 8, 16, out, None)
    assert e.value.status == sp.SP_EINVAL
    g.close()
    g_plain.close()
