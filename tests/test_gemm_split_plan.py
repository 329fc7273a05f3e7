"""Host logic of the tensor-core GEMM's split of a problem by its device-side live row count
(the prompt pass's mapper products): the plan for the model shapes, and its invariants over a
sweep (the narrow launch fits one wave up to m_split rows, the two launches' live-count ranges
cover every count once, the narrow width is half the bound's)."""
import ctypes

import pytest


@pytest.fixture(scope="module")
def lib():
    from paper_2601_03700_gb300 import build
    build.build()
    import paper_2601_03700_gb300 as adept
    L = adept.load_library()
    f = L.adept_debug_tc_split_plan
    f.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_int)]
    f.restype = ctypes.c_int
    return f


def plan(f, N, rows, sms=152):
    out = (ctypes.c_int * 3)()
    return tuple(out) if f(N, rows, sms, out) else None


def cdiv(a, b):
    return -(-a // b)


@pytest.mark.parametrize("N,rows,want", [
    (3072, 4096, (256, 128, 768)),    # GPT-2-small mapper FC1 / FC3, 8 x 512-token pass
    (6144, 4096, (256, 128, 384)),    # its FC2
    (768, 4096, (128, 64, 1536)),     # its FC4
    (8192, 2048, (256, 128, 256)),    # Llama-7B mapper FC1 / FC3, 2048-token pass
    (4096, 2048, (256, 128, 512)),    # its FC4
    (32768, 2048, None),              # its FC2: one row tile of 128-wide tiles exceeds a wave
    (1024, 64, None),                 # one row tile: nothing to split
    (512, 600, None),                 # the bound already takes the narrowest tiles
])
def test_plan_for_model_shapes(lib, N, rows, want):
    assert plan(lib, N, rows) == want


def test_plan_invariants(lib):
    for sms in (132, 148, 152):
        for N in (256, 512, 768, 1024, 2304, 3072, 4096, 6144, 8192, 11008, 16384, 32768):
            for rows in (129, 200, 256, 600, 1000, 2048, 4096, 8192):
                p = plan(lib, N, rows, sms)
                if p is None:
                    continue
                wide, narrow, m_split = p
                assert narrow * 2 == wide and narrow >= 32
                assert 128 <= m_split < rows and (m_split % 128 == 0 or m_split == rows - 1)
                # the narrow launch: one wave at m_split rows
                assert cdiv(m_split, 128) * cdiv(N, narrow) <= sms
                # the bound's width is the widest that gives every SM a tile at `rows`
                tm = cdiv(rows, 128)
                assert tm * cdiv(N, wide) >= sms
                if wide < 256:
                    assert tm * cdiv(N, wide * 2) < sms
