"""fxpq_fl_search_noalloc: the FL search for callers that cannot allocate device memory (a plug-in
whose host application owns the device memory pool, a loop that must never enter the allocator).
Its scratch is a static device array inside libfxpq.so, so it takes no workspace argument.

Checked through the C ABI against fxpq_fl_search with a caller workspace, on two calls in a row
with different inputs (the shared array keeps the previous call's contents, so the second call
also checks that the entry point clears it).  Same comparison as the other FL-search tests:
identical chosen FL and stats, scores within 1e-5 relative (and in fact identical)."""
import ctypes

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def test_noalloc_fl_search_matches_workspace_version_twice():
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import _lib as L
    lib = L.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    # the sorting kernel (k up to 16, k = 1 rows included) and the histogram kernel (k <= 8)
    cases = [("normal", 1 << 20, 2, -1, 2, 16, -8, 23), ("laplace", 300001, 3, 1, 4, 9, -2, 21),
             ("normal", 50000, 5, -1, 1, 16, -8, 23), ("relu_normal", 70001, 4, -1, 1, 8, -8, 23)]
    for dist, n, seed, S, klo, khi, fllo, flhi in cases:
        x = torch.from_numpy(synth.sweep_tensor(dist, n, seed)).cuda()
        nk, nfl = khi - klo + 1, flhi - fllo + 1
        outs = []
        for use_ws in (True, False):
            err = torch.full((nk * nfl,), -1.0, dtype=torch.float64, device="cuda")
            best = torch.full((nk,), -99, dtype=torch.int32, device="cuda")
            st = torch.zeros(ctypes.sizeof(L.Stats), dtype=torch.uint8, device="cuda")
            if use_ws:
                wsb = lib.fxpq_fl_search_workspace(n)
                ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
                rc = lib.fxpq_fl_search(_ptr(x), n, S, klo, khi, fllo, flhi, _ptr(err), _ptr(best), _ptr(st),
                                        _ptr(ws), wsb, stream)
            else:
                rc = lib.fxpq_fl_search_noalloc(_ptr(x), n, S, klo, khi, fllo, flhi, _ptr(err), _ptr(best), _ptr(st),
                                                stream)
            assert rc == L.OK
            torch.cuda.synchronize()
            outs.append((err.cpu().numpy(), best.cpu().numpy(), L.Stats.from_buffer_copy(bytes(st.cpu().numpy()))))
        (e1, b1, s1), (e2, b2, s2) = outs
        assert np.array_equal(b1, b2)
        np.testing.assert_allclose(e2, e1, rtol=1e-5, atol=0)
        assert np.array_equal(e2, e1)
        assert (s1.min, s1.max, s1.sum, s1.sumsq, s1.n, s1.is_signed) == (s2.min, s2.max, s2.sum, s2.sumsq, s2.n, s2.is_signed)
    assert lib.fxpq_get_device_status(stream) == L.OK


def test_noalloc_rejects_requests_beyond_its_limits():
    from paper_2203_12091_gb300 import _lib as L
    import __graft_entry__ as g
    g.build()
    lib = L.lib()
    p = ctypes.c_void_p(256)
    assert lib.fxpq_fl_search_noalloc(p, (1 << 31) + 1, -1, 2, 16, -8, 23, p, p, None, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search_noalloc(p, 100, -1, 2, 16, -8, 24, p, p, None, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search_noalloc(p, 100, -1, 2, 17, -8, 23, p, p, None, None) == L.ERR_INVALID_ARG
