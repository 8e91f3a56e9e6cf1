"""Coded-shuffling planner of libcm (host logic) against the oracle (Sec. IV).

The planner is C++ in the library; these tests need no GPU.  Partitions,
caches, the message plan of Alg. 1 and the layout of the received rows must
equal the oracle's exactly (the random draws follow one published
generator on both sides), and the realised rates must follow the theorem.
"""
import numpy as np
import pytest

import oracle.shuffle as osh


@pytest.fixture(scope="module")
def cm():
    import paper_1512_02673_gb300 as cm
    cm.lib()
    return cm


def _caches(S):
    owner, slots = S.caches()
    n = slots.shape[0]
    parts = [set(np.nonzero(owner == i)[0].tolist()) for i in range(n)]
    return parts, [set(slots[i].tolist()) for i in range(n)], slots


CASES = [(2, 40, 20), (3, 60, 20), (3, 60, 60), (4, 48, 30), (5, 50, 10), (6, 120, 47),
         (8, 64, 16), (4, 400, 170)]


@pytest.mark.parametrize("n,q,s", CASES)
def test_planner_equals_oracle(cm, n, q, s):
    lib = cm.Shuffle(n, q, s, 77, 88)
    sim = osh.Simulation(n, q, s, 77, 88)
    parts, caches, slots = _caches(lib)
    assert parts == sim.S and caches == sim.C
    assert all(len(set(slots[i].tolist())) == s for i in range(n))   # no slot twice
    for t in range(1, 5):
        st = lib.next()
        C0, S1 = sim.step()
        assert st["iteration"] == t
        parts, caches, slots = _caches(lib)
        assert parts == sim.S and caches == sim.C
        # Alg. 1: same messages, in the same order, with the same blocks
        A = {r: np.array([r], np.float64) for r in range(q)}
        msgs = osh.encode(C0, S1, A, "add")
        ptr, src, wk, sets = lib.plan()
        assert st["coded_rows"] == len(sets) == sum(m.shape[0] for _, _, m in msgs)
        assert st["message_sets"] == len(msgs)
        row = 0
        for I, blocks, msg in msgs:
            for j in range(msg.shape[0]):
                assert sets[row] == sum(1 << i for i in I)
                want = [(i, blocks[i][j]) for i in I if j < len(blocks[i])]
                got = list(zip(wk[ptr[row]:ptr[row + 1]].tolist(),
                               src[ptr[row]:ptr[row + 1]].tolist()))
                assert got == want
                row += 1
        # received rows: worker-major, ascending
        rptr, rrow = lib.received()
        coded, uncoded = osh.transition_counts(C0, S1)
        assert st["uncoded_rows"] == uncoded and st["coded_rows"] == coded
        for i in range(n):
            assert rrow[rptr[i]:rptr[i + 1]].tolist() == sorted(S1[i] - C0[i])
        # subtractions: every entry subtracts the other entries of its row
        counts = np.diff(ptr)
        assert st["subtractions"] == int(np.sum(counts * (counts - 1)))


def test_kept_rows_stay_in_their_slots(cm):
    n, q, s = 4, 200, 90
    lib = cm.Shuffle(n, q, s, 5, 6)
    _, _, before = _caches(lib)
    lib.next()
    _, after_sets, after = _caches(lib)
    rptr, rrow = lib.received()
    for i in range(n):
        new = set(rrow[rptr[i]:rptr[i + 1]].tolist())
        for c in range(s):
            if after[i, c] not in new:
                assert after[i, c] == before[i, c]


def test_rates_match_the_oracle_closed_form(cm):
    for n, q, s in [(50, 1000, 100), (8, 1e6, 2.5e5), (3, 300, 150), (16, 1e4, 1e4)]:
        rc, ru = cm.shuffle_rates(n, q, s)
        assert ru == pytest.approx(osh.uncoded_rate(q, s), rel=1e-14)
        assert rc == pytest.approx(osh.coded_rate(n, q, s), rel=1e-9, abs=1e-9 * q)
    rc, ru = cm.shuffle_rates(50, 1000, 100)
    assert 0.81 < 1 - rc / ru < 0.8105             # Sec. IV-D's printed reduction
    rc, ru = cm.shuffle_rates(10, 1000, 100)        # s = q/n
    assert rc == pytest.approx(ru / 2, rel=1e-14)


def test_realised_rates_follow_the_theorem_at_large_q(cm):
    # The uncoded count has expectation R_u exactly; the coded count tracks
    # R_c within ~1 %: the proof treats caches as independent, which the
    # update rule keeps only approximately (caches correlate slightly, and
    # the realised count settles a little below R_c).
    n, q, s = 4, 400000, 160000
    lib = cm.Shuffle(n, q, s, 1, 2)
    rc, ru = cm.shuffle_rates(n, q, s)
    for _ in range(6):
        st = lib.next()
        assert abs(st["uncoded_rows"] / ru - 1) < 0.005
        assert abs(st["coded_rows"] / rc - 1) < 0.02


@pytest.mark.parametrize("args", [(1, 10, 10), (3, 10, 5), (4, 40, 9), (4, 40, 41), (65, 130, 10),
                                  (4, 1 << 29, 1 << 27)])
def test_create_rejects_bad_shapes(cm, args):
    n, q, s = args
    with pytest.raises(cm.CodedError):
        cm.Shuffle(n, q, s, 1, 2)


def test_data_plane_needs_an_uploaded_plan(cm):
    # argument checks return before any device work: no GPU needed
    import ctypes
    lib = cm.Shuffle(3, 30, 15, 1, 2)
    L = cm.lib()
    nul = ctypes.c_void_p(0)
    assert L.cm_shuffle_encode(lib._h, nul, 0, nul, 4, 4, nul, 4, nul) == cm.CM_EINVAL
    assert L.cm_shuffle_fill(lib._h, nul, nul, 4, 4, nul, 4, nul) == cm.CM_EINVAL
    with pytest.raises(cm.CodedError):
        lib.plan()                         # no transition planned yet
    assert L.cm_shuffle_upload(lib._h, nul, 0, nul) == cm.CM_EINVAL
    assert lib.workspace_bytes() >= 4 * (30 * (3 + 5) + 3 * 15)


def test_device_planner_refuses_without_workspace(cm):
    # argument checks only (no GPU): device planning needs an initialised
    # workspace, and the dense set tables limit it to n <= 16
    import ctypes
    L = cm.lib()
    nul = ctypes.c_void_p(0)
    small = cm.Shuffle(4, 40, 20, 1, 2)
    assert L.cm_shuffle_device_next(small._h, nul, 0, nul, nul) == cm.CM_EINVAL
    assert L.cm_shuffle_device_init(small._h, nul, 0, nul) == cm.CM_EINVAL
    assert small.device_workspace_bytes() >= small.workspace_bytes()
    big = cm.Shuffle(17, 17 * 4, 8, 1, 2)
    assert big.device_workspace_bytes() == 0


@pytest.mark.parametrize("n,q,s", [(8, 1 << 16, 1 << 14), (4, 4000, 1700), (16, 3200, 800),
                                   (2, 40, 20)])
def test_device_workspace_size_formula(cm, n, q, s):
    # the size the header states for the device planner's workspace, to 10 %
    sh = cm.Shuffle(n, q, s, 1, 2)
    est = (sh.workspace_bytes() + 4 * q * (n + 21) + 4 * n * s + 16 * max(q, n * s)
           + 8 * n * 2 ** n + 2 ** 18 * n)
    got = sh.device_workspace_bytes()
    assert 0.9 * est <= got <= 1.1 * est, (got, est)
