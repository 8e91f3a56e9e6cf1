"""Coded shuffling data plane (Sec. IV) on the GPU against the oracle.

Every call goes through libcm's C ABI (``cm_shuffle_fill / encode / decode /
commit``).  Expected values come from ``oracle.shuffle``: its own partitions
and caches (same published generator and seeds), Alg. 1 over every worker
set, and decoding by subtraction, in exact arithmetic (fp64 for real sums,
integers for xor).

Tolerances.  xor is exact: bit-for-bit equality.  Real sums: a message row
sums e <= n fp32 rows left to right, so each element is within
(e-1) u sum_x |a_x| of the exact sum (u = 2^-24); a decoded row subtracts
e-1 cached rows from it, adding at most (e-1) u times the same magnitude
again, so |decoded - a| <= 2 (e-1) u sum_x |a_x|, plus the errors of the e-1
cached rows it subtracts, which carry earlier decodes (the test carries that
bound from transition to transition).
"""
import numpy as np
import pytest
import torch

import oracle.shuffle as osh
import synth

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24


@pytest.fixture(scope="module")
def cm():
    import paper_1512_02673_gb300 as cm
    cm.lib()
    return cm


def _padded(rows, r, dtype, dev="cuda"):
    """rows x r matrix whose leading dimension is a multiple of 4 words."""
    ld = (r + 3) // 4 * 4
    return torch.zeros((max(rows, 1), ld), dtype=dtype, device=dev)[:, :r]


def _oracle_messages(msgs, r, op):
    if not msgs:
        return np.zeros((0, r))
    return np.concatenate([m for _, _, m in msgs], axis=0)


def _oracle_received(n, msgs, C0, S1, A, op):
    rows = []
    for i in range(n):
        got = osh.decode(i, msgs, {x: A[x] for x in C0[i]}, op)
        for x in sorted(S1[i] - C0[i]):
            rows.append(got[x])
    return np.array(rows).reshape(len(rows), A.shape[1])


def _entry_magnitudes(msgs, A):
    """Per message row: (number of summed rows, elementwise sum of |a_x|)."""
    cnt, mag = [], []
    for _, blocks, m in msgs:
        for j in range(m.shape[0]):
            xs = [b[j] for b in blocks.values() if j < len(b)]
            cnt.append(len(xs))
            mag.append(np.sum(np.abs(A[xs].astype(np.float64)), axis=0))
    return np.array(cnt), np.array(mag).reshape(len(mag), A.shape[1])


@pytest.mark.parametrize("op", ["xor", "add"])
@pytest.mark.parametrize("n,q,s,r", [(4, 4000, 1700, 67), (3, 2400, 1200, 256),
                                     (5, 1500, 300, 1), (2, 1000, 700, 36)])
def test_transitions_match_oracle(cm, op, n, q, s, r):
    A32 = synth.gaussian((q, r), 1234 + r, "cpu").numpy()
    A = A32.view(np.uint32) if op == "xor" else A32
    dA = _padded(q, r, torch.float32)
    dA.copy_(torch.from_numpy(A32))
    lib = cm.Shuffle(n, q, s, 17, 19)
    sim = osh.Simulation(n, q, s, 17, 19)
    lib.upload()
    caches = lib.fill(dA, _padded(n * s, r, torch.float32))
    _, slots = lib.caches()
    torch.cuda.synchronize()
    assert torch.equal(caches, dA[torch.from_numpy(slots.reshape(-1)).long().cuda()])
    drift = np.zeros(r)
    for t in range(1, 4):
        st = lib.next()
        C0, S1 = sim.step()
        lib.upload()
        msgs = osh.encode(C0, S1, A, op)
        M = lib.encode(op, dA, _padded(st["coded_rows"], r, torch.float32))
        Rx = lib.decode(op, M, caches, r, _padded(st["uncoded_rows"], r, torch.float32))
        wantM = _oracle_messages(msgs, r, op)
        wantR = _oracle_received(n, msgs, C0, S1, A, op)
        gotM = M[:st["coded_rows"]].cpu().numpy()
        gotR = Rx[:st["uncoded_rows"]].cpu().numpy()
        if op == "xor":
            np.testing.assert_array_equal(gotM.view(np.uint32), wantM)
            np.testing.assert_array_equal(gotR.view(np.uint32), wantR)
        else:
            cnt, mag = _entry_magnitudes(msgs, A32)
            tolM = (cnt[:, None] - 1) * U32 * mag
            assert np.all(np.abs(gotM - wantM) <= tolM)
            # every received row: bound of its message row, doubled, plus drift
            ptr, src, wk, _ = lib.plan()
            rptr, rrow = lib.received()
            pos = {}
            for i in range(n):
                for u in range(rptr[i], rptr[i + 1]):
                    pos[(i, int(rrow[u]))] = u
            tolR = np.zeros_like(gotR)
            for m in range(len(ptr) - 1):
                for x in range(ptr[m], ptr[m + 1]):
                    # own rounding, plus the errors of the e-1 cached rows it subtracts
                    tolR[pos[(int(wk[x]), int(src[x]))]] = 2 * tolM[m] + (cnt[m] - 1) * drift
            assert np.all(np.abs(gotR - wantR) <= tolR)
            if len(tolR):
                drift = np.maximum(drift, np.max(tolR, axis=0))
        lib.commit(Rx, caches, r)
        _, slots = lib.caches()
        want_c = A32[slots.reshape(-1)]
        got_c = caches.cpu().numpy()
        if op == "xor":
            np.testing.assert_array_equal(got_c.view(np.uint32), want_c.view(np.uint32))
        else:
            assert np.all(np.abs(got_c - want_c) <= drift)


def test_edge_cases_nothing_to_send_and_pairs_only(cm):
    r = 32
    A = synth.gaussian((120, r), 5, "cuda")
    # s = q: every cache holds everything, no message
    lib = cm.Shuffle(4, 120, 120, 1, 2)
    lib.upload()
    caches = lib.fill(A)
    st = lib.next()
    assert st["coded_rows"] == 0 and st["uncoded_rows"] == 0
    lib.upload()
    M = lib.encode("xor", A)
    Rx = lib.decode("xor", M, caches, r)
    lib.commit(Rx, caches, r)
    _, slots = lib.caches()
    assert torch.equal(caches, A[torch.from_numpy(slots.reshape(-1)).long().cuda()])
    # s = q/n: caches hold only their sets; every message has |I| = 2
    lib = cm.Shuffle(4, 120, 30, 3, 4)
    lib.upload()
    caches = lib.fill(A)
    for _ in range(3):
        st = lib.next()
        _, _, _, sets = lib.plan()
        assert all(bin(int(x)).count("1") == 2 for x in sets)
        lib.upload()
        M = lib.encode("xor", A)
        Rx = lib.decode("xor", M, caches, r)
        lib.commit(Rx, caches, r)
        _, slots = lib.caches()
        assert torch.equal(caches, A[torch.from_numpy(slots.reshape(-1)).long().cuda()])


def test_stale_workspace_is_refused(cm):
    A = synth.gaussian((40, 8), 6, "cuda")
    lib = cm.Shuffle(2, 40, 30, 1, 2)
    lib.upload()
    caches = lib.fill(A)
    lib.next()
    with pytest.raises(cm.CodedError):
        lib.encode("xor", A)             # programs of the new transition not uploaded
    lib.upload()
    lib.encode("xor", A)


def test_real_sums_are_repeatable(cm):
    w = synth.SHUFFLE_SMALL
    A = _padded(w.q, w.r, torch.float32)
    A.copy_(synth.shuffle_rows(w, "cuda"))
    lib = cm.Shuffle(w.n, w.q, w.s, 8, 9)
    lib.upload()
    caches = lib.fill(A, _padded(w.n * w.s, w.r, torch.float32))
    st = lib.next()
    lib.upload()
    M1 = lib.encode("add", A, _padded(st["coded_rows"], w.r, torch.float32)).clone()
    M2 = lib.encode("add", A, _padded(st["coded_rows"], w.r, torch.float32))
    assert torch.equal(M1, M2)


def test_full_size_workload_by_properties(cm):
    # The data-plane workload the benchmark times, checked through properties
    # that hold at any size: after encode, decode and commit in xor every cache
    # slot holds exactly the data row its table names, and every received row
    # is exactly the data row the layout names; real sums stay within the
    # rounding bound.  Sampled message rows equal the xor of their rows.
    w = synth.SHUFFLE
    A = synth.shuffle_rows(w, "cuda")
    lib = cm.Shuffle(w.n, w.q, w.s, synth.SHUFFLE_PARTITION_SEED, synth.SHUFFLE_CACHE_SEED)
    lib.upload()
    caches = lib.fill(A)
    M = torch.empty((w.q, w.r), dtype=torch.float32, device="cuda")
    Rx = torch.empty((w.q, w.r), dtype=torch.float32, device="cuda")
    Ai = A.view(torch.int32)
    for t in range(2):
        st = lib.next()
        lib.upload()
        lib.encode("xor", A, M)
        lib.decode("xor", M, caches, w.r, Rx)
        rptr, rrow = lib.received()
        R = st["uncoded_rows"]
        assert torch.equal(Rx[:R], A[torch.from_numpy(rrow).long().cuda()])
        ptr, src, _, _ = lib.plan()
        rng = np.random.default_rng(t)
        for m in rng.integers(0, st["coded_rows"], 64):
            rows = torch.from_numpy(src[ptr[m]:ptr[m + 1]].astype(np.int64)).cuda()
            want = Ai[rows[0]].clone()
            for x in rows[1:]:
                want ^= Ai[x]
            assert torch.equal(M[m].view(torch.int32), want)
        lib.commit(Rx, caches, w.r)
        _, slots = lib.caches()
        assert torch.equal(caches, A[torch.from_numpy(slots.reshape(-1)).long().cuda()])
    # one transition in real arithmetic on the same state
    st = lib.next()
    lib.upload()
    lib.encode("add", A, M)
    lib.decode("add", M, caches, w.r, Rx)
    _, rrow = lib.received()
    R = st["uncoded_rows"]
    exact = A[torch.from_numpy(rrow).long().cuda()]
    # at most n rows of magnitude <= max|a| per message row, caches exact
    err = (Rx[:R] - exact).abs().max().item()
    assert err <= 2 * (w.n - 1) * U32 * w.n * A.abs().max().item()
