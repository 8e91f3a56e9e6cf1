"""Host-side tests of libcm: no GPU needed, no kernel launched.

The library loads on a machine without a GPU (the CUDA runtime is linked
statically); these tests call only its host logic: symbol exports, the
straggler draw (bit-exact against the oracle's independent implementation),
code construction and the synchronous argument checks that run before any
launch.
"""
import ctypes
import os
import re

import numpy as np
import pytest

import synth
from conftest import ROOT


@pytest.fixture(scope="session")
def cm():
    from paper_1512_02673_gb300 import build
    import paper_1512_02673_gb300 as cm
    if not os.path.exists(cm.LIB_PATH):
        build.build()
    cm.lib()
    return cm


def declared_functions():
    src = open(os.path.join(ROOT, "include", "cm.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(cm_[a-z0-9_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(cm):
    names = declared_functions()
    assert len(names) >= 13, names
    lib = ctypes.CDLL(cm.LIB_PATH)
    for name in names:
        assert hasattr(lib, name), name


def test_status_strings(cm):
    for s in range(0, -8, -1):
        assert cm.status_string(s) and "unknown" not in cm.status_string(s)
    assert "unknown" in cm.status_string(-99)


@pytest.mark.parametrize("n,k", [(6, 3), (10, 5), (20, 10), (32, 24), (16, 12), (3, 2),
                                 (32, 1), (32, 31), (2, 1)])
def test_erasure_draw_is_bit_exact_with_oracle(cm, orc, n, k):
    for seed in (synth.ERASURE_SEED, 0, 2**64 - 1, 0x123456789ABCDEF):
        for counter in list(range(60)) + [2**40, 2**63]:
            m1, t1 = cm.draw_erasures(seed, counter, n, k)
            m2, t2 = orc.draw_erasures(seed, counter, n, k)
            assert m1 == m2, (seed, counter)
            np.testing.assert_allclose(t1, t2, rtol=1e-15, atol=0)


def test_erasure_draw_shape_parameters(cm):
    # the ranking does not depend on shift / rate; the times do
    m1, t1 = cm.draw_erasures(9, 4, 10, 5, shift=1.0, rate=1.0)
    m2, t2 = cm.draw_erasures(9, 4, 10, 5, shift=3.0, rate=0.25)
    assert m1 == m2
    np.testing.assert_allclose((t2 * 5 - 3.0) * 0.25, t1 * 5 - 1.0, rtol=1e-12)


def test_erasure_draw_rejects_bad_arguments(cm):
    for args in [(0, 1), (33, 3), (5, 0), (5, 6)]:
        with pytest.raises(cm.CodedError):
            cm.draw_erasures(1, 0, *args)
    with pytest.raises(cm.CodedError):
        cm.draw_erasures(1, 0, 6, 3, rate=0.0)


def test_code_construction(cm):
    P = synth.parity_coefficients(32, 24)
    c = cm.Code(32, 24, 65536, 65536, P)
    assert c.L == 2731
    assert cm.Code(6, 3, 1200, 500, synth.parity_coefficients(6, 3)).L == 400
    for bad in [(3, 3, 10, 10), (33, 3, 10, 10), (6, 0, 10, 10), (6, 3, 0, 10), (6, 3, 10, 0)]:
        n, k = bad[0], bad[1]
        with pytest.raises((cm.CodedError, ValueError)):
            cm.Code(*bad, np.zeros((max(n - k, 1), max(k, 1)), np.float32))
    Pn = P.copy()
    Pn[0, 0] = np.nan
    with pytest.raises(cm.CodedError):
        cm.Code(32, 24, 100, 100, Pn)


def test_synchronous_checks_precede_any_launch(cm):
    """Rejected calls return before touching the device (safe without a GPU)."""
    L = cm.lib()
    c = cm.Code(6, 3, 1200, 500, synth.parity_coefficients(6, 3))
    fake = ctypes.c_void_p(1 << 20)     # never dereferenced: every call below is rejected
    # fewer than k survivors
    assert L.cm_decode(c.handle, fake, 0b000011, 1, fake, None, None) == cm.CM_ENOTDECODABLE
    # survivor bit at or above n
    assert L.cm_decode(c.handle, fake, 0b1000111, 1, fake, None, None) == cm.CM_EINVAL
    # b out of range, misaligned operands, bad leading dimension
    assert L.cm_matvec(c.handle, fake, 500, fake, 500, fake, 9, fake, None, None) == cm.CM_EINVAL
    assert L.cm_matvec(c.handle, fake, 500, fake, 500, fake, 0, fake, None, None) == cm.CM_EINVAL
    odd = ctypes.c_void_p((1 << 20) + 4)
    assert L.cm_matvec(c.handle, odd, 500, fake, 500, fake, 1, fake, None, None) == cm.CM_EINVAL
    assert L.cm_matvec(c.handle, fake, 501, fake, 500, fake, 1, fake, None, None) == cm.CM_EINVAL
    assert L.cm_matvec(c.handle, fake, 496, fake, 500, fake, 1, fake, None, None) == cm.CM_EINVAL
    assert L.cm_encode(c.handle, fake, 502, fake, 500, None, None) == cm.CM_EINVAL
    assert L.cm_encode(None, fake, 500, fake, 500, None, None) == cm.CM_EINVAL
    # f32 code refuses the bf16-only tensor-core path
    assert L.cm_coded_gemm(c.handle, fake, 512, fake, 512, fake, 512, 64, fake, 64,
                           None, None) == cm.CM_EINVAL
    cb = cm.Code(6, 3, 120, 64, synth.parity_coefficients(6, 3), dtype="bf16")
    assert L.cm_coded_gemm(cb.handle, fake, 64, fake, 64, fake, 64, 0, fake, 24,
                           None, None) == cm.CM_EINVAL    # N < 1
    assert L.cm_coded_gemm(cb.handle, fake, 68, fake, 64, fake, 64, 32, fake, 32,
                           None, None) == cm.CM_EINVAL    # lda not 16-byte pitched
    assert L.cm_matvec(cb.handle, fake, 64, fake, 64, fake, 1, fake, None, None) == cm.CM_EINVAL
    # survivors-only GEMM: the survivor checks come before any launch
    assert L.cm_coded_gemm_survivors(cb.handle, fake, 64, fake, 64, fake, 64, 32, 0b000011,
                                     fake, 32, None, None) == cm.CM_ENOTDECODABLE
    assert L.cm_coded_gemm_survivors(cb.handle, fake, 64, fake, 64, fake, 64, 32, 0b1000111,
                                     fake, 32, None, None) == cm.CM_EINVAL
    assert L.cm_coded_gemm_survivors(c.handle, fake, 512, fake, 512, fake, 512, 32, 0b111,
                                     fake, 32, None, None) == cm.CM_EINVAL   # f32 code
    assert L.cm_coded_gemm_survivors(cb.handle, fake, 64, fake, 64, fake, 64, 32, 0b111,
                                     fake, 24, None, None) == cm.CM_EINVAL   # ldc < N


def test_gd_workspace_and_checks(cm):
    L = cm.lib()
    m, d = 400, 80
    cA = cm.Code(20, 10, m, d, synth.parity_coefficients(20, 10))
    cAT = cm.Code(20, 10, d, m, synth.parity_coefficients(20, 10, seed=synth.CODE_SEED + 1))
    ws = cm.gd_workspace_bytes(cA, cAT)
    assert ws >= 8 * 20 * cA.L + 4 * m + 8 * 20 * cAT.L
    assert ws % 256 == 0
    fake = ctypes.c_void_p(1 << 20)
    full = (1 << 20) - 1
    # too small a workspace
    assert L.cm_gd_step(cA.handle, fake, d, fake, d, cAT.handle, fake, m, fake, m, fake, fake,
                        0.1, full, full, fake, ws - 1, None, None) == cm.CM_ENOMEM
    # codes that are not transposes of each other
    assert L.cm_gd_step(cA.handle, fake, d, fake, d, cA.handle, fake, d, fake, d, fake, fake,
                        0.1, full, full, fake, ws, None, None) == cm.CM_EINVAL
    # a product with fewer than k survivors
    assert L.cm_gd_step(cA.handle, fake, d, fake, d, cAT.handle, fake, m, fake, m, fake, fake,
                        0.1, 0b111, full, fake, ws, None, None) == cm.CM_ENOTDECODABLE


def test_static_scratch_size_matches_header(cm):
    # The binding's copy of CM_GD_STATIC_SCRATCH_BYTES is the header's value.
    src = open(os.path.join(ROOT, "include", "cm.h")).read()
    m = re.search(r"#define\s+CM_GD_STATIC_SCRATCH_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", src)
    assert m, "CM_GD_STATIC_SCRATCH_BYTES not found in cm.h"
    assert cm.GD_STATIC_SCRATCH_BYTES == int(m.group(1)) << int(m.group(2))
