"""The retrieval for callers that cannot allocate device memory: crc_retrieve_noalloc.

Some callers of this library cannot allocate GPU memory while they run: an engine's
render thread with a fixed per-frame budget (cudaMalloc and cudaFree can synchronise
the device), a plugin whose host application owns all GPU memory, a stream that must
not fail half-way with an out-of-memory error.  crc_retrieve_noalloc serves them with
a fixed scratch array inside the library instead of a caller workspace.

The GPU test calls it through the C ABI and checks it against crc_retrieve with a
caller workspace on two calls in a row (the shared scratch keeps the first call's
contents): identical indices, scores and counts, and identical gathered keys and
values (retrieval results are bit-exact, the tolerance the other retrieval tests use).
This file is collected last, so that a run stopping at the first failure has run
every other test before it.
"""

import ctypes as C
import math

import numpy as np
import pytest

from paper_2607_21848_gb300 import _abi


@pytest.fixture(scope="module")
def lib():
    from paper_2607_21848_gb300 import build
    build.build()
    return _abi.load()


def _frames(F, pos, yaw):
    fr = (_abi.crc_frame * F)()
    c, s = math.cos(yaw), math.sin(yaw)
    # camera-to-world rotation whose third column (the optical axis) points along (c, s, 0)
    R = [s, 0.0, c, -c, 0.0, s, 0.0, -1.0, 0.0]
    for f in range(F):
        fr[f].K[:] = [4.0, 0.0, 3.5, 0.0, 4.0, 3.5, 0.0, 0.0, 1.0]
        fr[f].R[:] = R
        fr[f].c[:] = [pos[0], pos[1], 1.6 + 0.01 * f]
    return fr


def test_noalloc_rejects_banks_beyond_its_scratch(lib):
    """Checked on the host before any CUDA call: a bank whose candidates would not fit the
    fixed scratch is refused with its own status code."""
    F = 2
    shape = _abi.crc_shape(1, 1, 64, F, 8, 8, _abi.CRC_F32)
    fake = 1 << 20
    B = 300000
    bank = _abi.crc_bank(B, 1, fake, fake, fake, fake, fake, None)
    params = _abi.crc_retrieval(1.0, 0.5, math.inf, -1.0, 1, 8, -1, 0, 0)
    assert lib.crc_retrieve_workspace_size(B, 8) > _abi.CRC_NOALLOC_SCRATCH_BYTES
    st = lib.crc_retrieve_noalloc(C.byref(bank), B, C.byref(shape), _frames(F, (0, 0), 0.0), B, C.byref(params),
                                  None, None, fake, None, fake, None)
    assert st == _abi.CRC_ERR_TOO_LARGE
    assert b"fixed scratch" in lib.crc_status_string(st)
    assert lib.crc_retrieve_noalloc(C.byref(bank), B, C.byref(shape), _frames(F, (0, 0), 0.0), B, None, None, None,
                                    fake, None, fake, None) == _abi.CRC_ERR_INVALID_ARG
    # at k = 1 every bank fits
    assert lib.crc_retrieve_workspace_size(B, 1) <= _abi.CRC_NOALLOC_SCRATCH_BYTES


@pytest.mark.gpu
def test_noalloc_matches_the_workspace_call_on_two_calls_in_a_row(lib):
    import torch

    from paper_2607_21848_gb300 import api

    F, h, w, L, H, d, k, B, P = 2, 8, 8, 1, 2, 64, 8, 20000, 4
    Nc = F * h * w
    shape = api.shape(L, H, d, F, h, w, torch.float32)
    g = np.random.default_rng(5)
    bank = api.Bank(B, F, h, w, L, H, d, torch.float32, P)
    c = g.normal(size=(B, 3)) * 20.0
    v = g.normal(size=(B, 3))
    v /= np.linalg.norm(v, axis=1, keepdims=True)
    bank.centre.copy_(torch.from_numpy(c))
    bank.view.copy_(torch.from_numpy(v))
    bank.kv.copy_(torch.randn(bank.kv.shape, generator=torch.Generator().manual_seed(6)))
    need = lib.crc_retrieve_workspace_size(B, k)
    assert 0 < need <= _abi.CRC_NOALLOC_SCRATCH_BYTES  # several blocks: the scratch is in use
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    segs = [(0, Nc, api.SEG_SINK, 0)] + [((1 + r) * Nc, Nc, api.SEG_RETRIEVED, r) for r in range(k)]
    params = _abi.crc_retrieval(10.0, 0.5, math.inf, -1.0, 1, k, -1, 0, 0)
    bs, sh = bank.struct(), shape
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)

    def run(noalloc, pos, yaw):
        cache = api.Cache.empty(L, (1 + k) * Nc, H, d, torch.float32, segs)
        idx = torch.full((k,), -7, dtype=torch.int32, device="cuda")
        score = torch.full((k,), -7.0, dtype=torch.float64, device="cuda")
        count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
        cs = cache.struct()
        fr = _frames(F, pos, yaw)
        if noalloc:
            st = lib.crc_retrieve_noalloc(C.byref(bs), B, C.byref(sh), fr, B, C.byref(params), C.byref(cs), None,
                                          idx.data_ptr(), score.data_ptr(), count.data_ptr(), stream)
        else:
            st = lib.crc_retrieve(C.byref(bs), B, C.byref(sh), fr, B, C.byref(params), C.byref(cs), None,
                                  idx.data_ptr(), score.data_ptr(), count.data_ptr(), ws.data_ptr(), need, stream)
        assert st == _abi.CRC_OK
        torch.cuda.synchronize()
        return idx.cpu(), score.cpu(), count.cpu(), cache.k.cpu(), cache.v.cpu()

    poses = [((3.0, -2.0), 0.3), ((-11.0, 7.5), 2.2)]
    for pos, yaw in poses:  # two calls in a row through the shared scratch
        got = run(True, pos, yaw)
        ref = run(False, pos, yaw)
        assert int(ref[2]) == k
        for a, b in zip(got, ref):
            assert torch.equal(a, b)
    # the two poses retrieve different chunks, so the second call did not reuse the first's result
    assert not torch.equal(run(True, *poses[0])[0], run(True, *poses[1])[0])
