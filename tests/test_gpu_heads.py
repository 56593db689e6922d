"""Head sharding (Sec. 4.3: attention heads are independent, Eq. 2 acts per head).

A deployment over several GPUs gives each GPU a range of heads: its own K/V slab pool
for those heads, and strided views of the queries, cache and outputs (the base pointer
moved by h0 * d, H/2 heads, the full tensor's strides).  The reprojection is per query
and head-free, so every GPU computes it.  Here two head halves, each run through the
C ABI on such views, must reproduce the full call bit for bit: the cache update, the
retrieval's gather and the biased attention."""

import numpy as np
import pytest
import torch

import synth
from paper_2607_21848_gb300 import api

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_21848_gb300 import build
    build.build()


def test_two_head_halves_reproduce_the_full_call_bit_for_bit():
    wl = synth.make_workload(2, layers=2, heads=4, bank=16, grid=(12, 16))
    L, H, d, F, h, w, k = wl.L, wl.H, wl.d, wl.F, wl.h, wl.w, wl.k
    Nc = F * h * w
    g = torch.Generator(device="cuda").manual_seed(31)

    def rnd(*shape):
        return (torch.randn(*shape, generator=g, device="cuda") * wl.qkv_scale).bfloat16()

    pool = rnd(wl.num_slabs, 2, L, Nc, H, d)
    cache_init = (rnd(L, wl.n_keys, H, d), rnd(L, wl.n_keys, H, d))
    q = rnd(L, Nc, H, d)
    k_new, v_new = rnd(L, Nc, H, d), rnd(L, Nc, H, d)
    depth = torch.from_numpy(wl.depth_of(wl.n)).cuda()
    frames = synth.frame_records(wl.cur_frames)
    win_off = [off for off, _, kind, _ in wl.segments if kind == api.SEG_WINDOW][-1]
    params = api.retrieval_params(wl.E, wl.w_v, wl.tau_c, wl.cos_tau_v, wl.delta, k)

    def bank_for(heads):
        b = api.Bank(wl.bank_size + 1, F, h, w, L, len(heads), d, torch.bfloat16, wl.num_slabs)  # + chunk n
        api.crc_bank_insert_poses(b, api.shape(L, len(heads), d, F, h, w, torch.bfloat16), 0,
                                  synth.frame_records(wl.bank_frames))
        b.depth[:wl.bank_size].copy_(torch.from_numpy(wl.depth_bank()).cuda())
        b.kv.copy_(pool[..., heads, :])
        return b

    def step(cache, qv, o, heads, full_shape):
        shp = api.shape(L, len(heads), d, F, h, w, torch.bfloat16)
        bank = bank_for(heads)
        idx = torch.zeros(k, dtype=torch.int32, device="cuda")
        cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
        uv = torch.zeros(Nc, k * F, 2, device="cuda")
        valid = torch.zeros(Nc, k * F, dtype=torch.uint8, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        kn = k_new[:, :, heads].contiguous()
        vn = v_new[:, :, heads].contiguous()
        api.crc_cache_update(bank, shp, wl.n, frames, depth, kn, vn, cache, win_off)
        api.crc_retrieve(bank, wl.bank_size, shp, frames, wl.n, params, cache, idx, None, cnt)
        api.crc_correspond(shp, frames, depth, bank, idx, cnt, k, wl.eps, uv, None, valid)
        api.crc_biased_attention(shp, qv, cache, o, None, uv, valid, k, idx, wl.lam, wl.sigma, 0, status)
        torch.cuda.synchronize()
        assert status.item() == 0
        return idx, uv, valid, bank

    # the full call over all heads
    full = api.Cache(cache_init[0].clone(), cache_init[1].clone(), wl.segments)
    o_full = torch.full_like(q, float("nan"))
    idx_f, uv_f, valid_f, bank_f = step(full, q, o_full, list(range(H)), True)
    # two halves on head views of one shared cache, query and output
    shared = api.Cache(cache_init[0].clone(), cache_init[1].clone(), wl.segments)
    o_half = torch.full_like(q, float("nan"))
    for rank in range(2):
        h0, nh = api.head_range(H, rank, 2)
        heads = list(range(h0, h0 + nh))
        view = shared.heads(h0, nh)
        assert view.k.data_ptr() == shared.k.data_ptr() + h0 * d * 2 and view.k.stride() == shared.k.stride()
        idx_h, uv_h, valid_h, bank_h = step(view, api.head_view(q, h0, nh), api.head_view(o_half, h0, nh), heads,
                                            False)
        assert torch.equal(idx_h, idx_f) and torch.equal(valid_h, valid_f)
        assert torch.equal(uv_h.view(torch.int32), uv_f.view(torch.int32))
        assert torch.equal(bank_h.kv, bank_f.kv[..., heads, :])  # the new chunk's slab, per half
    assert int(idx_f[0]) >= 0 and bool(valid_f.any())  # a retrieval with correspondences took place
    assert torch.equal(shared.k, full.k) and torch.equal(shared.v, full.v)  # window write and gather
    assert torch.equal(o_half, o_full)  # attention, every head
