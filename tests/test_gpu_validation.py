"""Host-side validation of every entry point: each bad argument is rejected with its
documented status code before anything is enqueued (outputs keep their sentinel
values).  Fault injection for this library happens here, on the host: nothing in
these tests reaches a kernel with an invalid argument."""

import math

import numpy as np
import pytest
import torch

import synth
from paper_2607_21848_gb300 import _abi, api
from tests import _gpu

pytestmark = pytest.mark.gpu

INVALID, SHAPE, UNSUPPORTED = _abi.CRC_ERR_INVALID_ARG, _abi.CRC_ERR_SHAPE, _abi.CRC_ERR_UNSUPPORTED


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_21848_gb300 import build
    build.build()


def _status(fn, *args, **kw):
    with pytest.raises(api.CrcError) as e:
        fn(*args, **kw)
    torch.cuda.synchronize()
    return e.value.status


@pytest.fixture(scope="module")
def small():
    wl = synth.make_workload(2, layers=1, heads=2, bank=8, grid=(8, 16))
    shp = api.shape(wl.L, wl.H, wl.d, wl.F, wl.h, wl.w, torch.bfloat16)
    bank = api.Bank(8, wl.F, wl.h, wl.w, wl.L, wl.H, wl.d, torch.bfloat16, 4)
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    Nc = wl.Nc
    segs = [(0, Nc, api.SEG_SINK, 0), (Nc, Nc, api.SEG_RETRIEVED, 0), (2 * Nc, 2 * Nc, api.SEG_WINDOW, 0)]
    cache = api.Cache.empty(wl.L, 4 * Nc, wl.H, wl.d, torch.bfloat16, segs)
    return wl, shp, bank, cache


def test_insert_poses_rejections(small):
    wl, shp, bank, _ = small
    rec = synth.frame_records(wl.bank_frames[:1])
    assert _status(api.crc_bank_insert_poses, bank, shp, 8, rec) == INVALID  # first + count > capacity
    bad = rec.copy()
    bad[0, 0] = math.nan  # non-finite intrinsics
    assert _status(api.crc_bank_insert_poses, bank, shp, 0, bad) == INVALID
    bad = rec.copy()
    bad[0, 8] = 2.0  # K's last row must be (0, 0, 1)
    assert _status(api.crc_bank_insert_poses, bank, shp, 0, bad) == INVALID


def test_cache_update_rejections(small):
    wl, shp, bank, cache = small
    fr = synth.frame_records(wl.bank_frames[0])
    depth = torch.ones(wl.F, wl.h, wl.w, device="cuda")
    k = torch.zeros(wl.L, wl.Nc, wl.H, wl.d, dtype=torch.bfloat16, device="cuda")
    before = cache.k.clone()
    assert _status(api.crc_cache_update, bank, shp, 8, fr, depth, k, k, cache, 0) == INVALID  # chunk >= capacity
    assert _status(api.crc_cache_update, bank, shp, 1, fr, depth, k, None, cache, 0) == INVALID  # K without V
    assert _status(api.crc_cache_update, bank, shp, 1, fr, depth, k, k, cache, 3 * wl.Nc + 1) == SHAPE
    flat = torch.zeros(k.numel() + 8, dtype=torch.bfloat16, device="cuda")
    k_mis = flat[1:1 + k.numel()].view(k.shape)  # 2-byte offset: not 16-byte aligned
    assert _status(api.crc_cache_update, bank, shp, 1, fr, depth, k_mis, k, cache, 0) == UNSUPPORTED
    assert torch.equal(before, cache.k)


def test_retrieve_and_gather_rejections(small):
    wl, shp, bank, cache = small
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    count = torch.zeros(1, dtype=torch.int32, device="cuda")
    cur = synth.frame_records(wl.bank_frames[3])
    for params in (api.retrieval_params(0.0, 0.5, 1.0, -1.0, 1, 1),          # E must be > 0
                   api.retrieval_params(1.0, 0.5, 1.0, -1.0, 1, 0),          # k in 1..8
                   api.retrieval_params(1.0, 0.5, 1.0, -1.0, 1, 9),
                   api.retrieval_params(1.0, math.nan, 1.0, -1.0, 1, 1)):    # NaN weight
        assert _status(api.crc_retrieve, bank, 8, shp, cur, 3, params, cache, idx, None, count) == INVALID
    ok = api.retrieval_params(1.0, 0.5, 1.0, -1.0, 1, 1)
    assert _status(api.crc_retrieve, bank, 9, shp, cur, 3, ok, cache, idx, None, count) == INVALID  # > capacity
    # two retrieved segments claiming the same slot
    Nc = wl.Nc
    dup = api.Cache(cache.k, cache.v, [(0, Nc, api.SEG_RETRIEVED, 0), (Nc, Nc, api.SEG_RETRIEVED, 0)])
    assert _status(api.crc_retrieve, bank, 8, shp, cur, 3, ok, dup, idx, None, count) == SHAPE
    assert _status(api.crc_gather, shp, bank.kv, idx, 1, dup) == SHAPE


def test_correspond_rejections(small):
    wl, shp, bank, _ = small
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    depth = torch.ones(wl.F, wl.h, wl.w, device="cuda")
    S = wl.F
    uv = torch.full((wl.Nc, S, 2), -9.0, device="cuda")
    valid = torch.full((wl.Nc, S), 9, dtype=torch.uint8, device="cuda")
    cur = synth.frame_records(wl.bank_frames[3])
    for k, eps in ((0, 0.05), (9, 0.05), (1, -0.1), (1, math.nan)):
        assert _status(api.crc_correspond, shp, cur, depth, bank, idx, None, k, eps, uv, None, valid) == INVALID
    flat = torch.zeros(uv.numel() + 2, device="cuda")
    uv_mis = flat[1:1 + uv.numel()].view(uv.shape)  # 4-byte offset: float2 stores need 8
    assert _status(api.crc_correspond, shp, cur, depth, bank, idx, None, 1, 0.05, uv_mis, None, valid) == UNSUPPORTED
    assert bool((uv == -9.0).all()) and bool((valid == 9).all())


def test_attention_rejections(small):
    wl, shp, bank, cache = small
    q = torch.zeros(wl.L, wl.Nc, wl.H, wl.d, dtype=torch.bfloat16, device="cuda")
    o = torch.full_like(q, 7.0)
    S = wl.F
    uv = torch.zeros(wl.Nc, S, 2, device="cuda")
    valid = torch.zeros(wl.Nc, S, dtype=torch.uint8, device="cuda")
    att = api.crc_biased_attention
    assert _status(att, shp, q[:, :-8], cache, o[:, :-8], None, uv, valid, 1, None, 2.0, 1.0) == SHAPE  # n_q != N_c
    assert _status(att, shp, q, cache, o, None, uv, valid, 1, None, -1.0, 1.0) == INVALID  # lambda < 0
    assert _status(att, shp, q, cache, o, None, uv, valid, 1, None, 2.0, 0.0) == INVALID  # sigma = 0
    assert _status(att, shp, q, cache, o, None, None, None, 1, None, 2.0, 1.0) == INVALID  # no correspondences
    assert _status(att, shp, q, cache, o, None, uv, valid, 0, None, 2.0, 1.0) == SHAPE  # retrieved slot >= k
    Nc = wl.Nc
    overlap = api.Cache(cache.k, cache.v, [(0, 2 * Nc, api.SEG_SINK, 0), (Nc, Nc, api.SEG_WINDOW, 0)])
    assert _status(att, shp, q, overlap, o, None, uv, valid, 1, None, 2.0, 1.0) == SHAPE
    badkind = api.Cache(cache.k, cache.v, [(0, Nc, 7, 0)])
    assert _status(att, shp, q, badkind, o, None, uv, valid, 1, None, 2.0, 1.0) == INVALID
    # bf16 with d = 64 is not a tensor-core shape; the SIMT kernel takes it
    shp64 = api.shape(wl.L, wl.H, 64, wl.F, wl.h, wl.w, torch.bfloat16)
    c64 = api.Cache.empty(wl.L, 4 * Nc, wl.H, 64, torch.bfloat16, cache.segments)
    q64 = torch.zeros(wl.L, Nc, wl.H, 64, dtype=torch.bfloat16, device="cuda")
    o64 = torch.full_like(q64, 7.0)
    assert _status(att, shp64, q64, c64, o64, None, uv, valid, 1, None, 2.0, 1.0) == UNSUPPORTED
    att(shp64, q64, c64, o64, None, uv, valid, 1, None, 2.0, 1.0, flags=api.ATTN_SIMT)
    torch.cuda.synchronize()
    assert bool((o64 == 0).all())  # zero values everywhere: the output is zero
    assert bool((o == 7.0).all())  # none of the rejected calls wrote the output
