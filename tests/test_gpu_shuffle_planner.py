"""The coded-shuffling planner on the device against the host planner (Sec. IV).

Two instances with the same seeds: one planned on the host (cm_shuffle_next,
itself pinned to the oracle in tests/test_shuffle_host.py), one on the device
(cm_shuffle_device_next).  Every transition must give the same plan bit for
bit: counts, message plan, received layout, partition, slot tables and the
row programs in the workspace.  Then the data plane runs on the
device-planned workspace and every cache slot must hold exactly its row.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cm():
    import paper_1512_02673_gb300 as cm
    cm.lib()
    return cm


def _words(ws, off, count):
    """count int32 words of a device workspace starting at word off."""
    if count == 0:
        return np.zeros(0, np.int32)
    return ws.view(torch.int32)[off:off + count].cpu().numpy()


def _layout(n, q, s):
    """Word offsets of the row programs (the layout of cm_shuffle_upload)."""
    up = lambda x: (x + 63) & ~63
    L, at = {}, 0
    for name, size in [("enc_ptr", q + 1), ("enc_src", q), ("dec_msg", q), ("dec_ptr", q + 1),
                       ("dec_slot", q * (n - 1)), ("dec_dst", q), ("com_dst", q),
                       ("fill_row", n * s)]:
        L[name] = at
        at += up(size)
    return L


def _same_plan(cm, h, d, n, q, s):
    for a, b in zip(h.plan(), d.plan()):
        np.testing.assert_array_equal(a, b)
    for a, b in zip(h.received(), d.received()):
        np.testing.assert_array_equal(a, b)
    for a, b in zip(h.caches(), d.caches()):
        np.testing.assert_array_equal(a, b)
    st = h.stats()
    C, R, X = st["coded_rows"], st["uncoded_rows"], st["subtractions"]
    L = _layout(n, q, s)
    for name, count in [("enc_ptr", C + 1), ("enc_src", R), ("dec_msg", R), ("dec_ptr", R + 1),
                        ("dec_slot", X), ("dec_dst", R), ("com_dst", R), ("fill_row", n * s)]:
        np.testing.assert_array_equal(_words(h._ws, L[name], count),
                                      _words(d._ws, L[name], count), err_msg=name)


@pytest.mark.parametrize("n,q,s", [(2, 40, 20), (3, 600, 300), (4, 4000, 1700), (5, 1500, 300),
                                   (8, 8000, 2000), (4, 120, 120), (16, 3200, 800),
                                   (6, 6000, 2500),
                                   (4, 400, 100),    # s = q/n: the cache keeps no candidate
                                   (16, 32, 3)])     # q/n = 2: most partition buckets straddle
def test_device_plans_equal_host_plans(cm, n, q, s):
    h = cm.Shuffle(n, q, s, 23, 29)
    d = cm.Shuffle(n, q, s, 23, 29)
    h.upload()
    d.device_init()
    for t in range(1, 5):
        sh = h.next()
        h.upload()
        sd = d.device_next()
        assert sh == sd
        _same_plan(cm, h, d, n, q, s)


def test_device_init_after_host_transitions(cm):
    # switching to the device after two host-planned transitions keeps the
    # current programs and continues the same sequence
    n, q, s = 4, 2000, 900
    h = cm.Shuffle(n, q, s, 5, 6)
    d = cm.Shuffle(n, q, s, 5, 6)
    for _ in range(2):
        h.next()
        d.next()
    h.upload()
    d.device_init()
    _same_plan(cm, h, d, n, q, s)
    for _ in range(2):
        assert h.next() == d.device_next()
        h.upload()
        _same_plan(cm, h, d, n, q, s)
    with pytest.raises(cm.CodedError):
        d.next()                      # device-mode instances plan on the device
    with pytest.raises(cm.CodedError):
        d.upload()


def test_data_plane_on_device_plans(cm):
    n, q, s, r = 8, 20000, 5000, 64
    A = synth.gaussian((q, r), 77, "cuda")
    d = cm.Shuffle(n, q, s, 3, 4)
    d.device_init()
    caches = d.fill(A)
    for _ in range(3):
        st = d.device_next()
        M = d.encode("xor", A)
        Rx = d.decode("xor", M, caches, r)
        _, rrow = d.received()
        assert torch.equal(Rx[:st["uncoded_rows"]], A[torch.from_numpy(rrow).long().cuda()])
        d.commit(Rx, caches, r)
        _, slots = d.caches()
        assert torch.equal(caches, A[torch.from_numpy(slots.reshape(-1)).long().cuda()])


def test_full_size_device_plan_equals_host(cm):
    w = synth.SHUFFLE
    h = cm.Shuffle(w.n, w.q, w.s, synth.SHUFFLE_PARTITION_SEED, synth.SHUFFLE_CACHE_SEED)
    d = cm.Shuffle(w.n, w.q, w.s, synth.SHUFFLE_PARTITION_SEED, synth.SHUFFLE_CACHE_SEED)
    h.upload()
    d.device_init()
    for _ in range(2):
        assert h.next() == d.device_next()
        h.upload()
        _same_plan(cm, h, d, w.n, w.q, w.s)
