"""GPU parity of the mirror gather (crc_gather) and of the RoPE re-positioning of
re-packed keys (Sec. 4.2 "Cache packing") against the oracle.

Plain gathers are byte-exact.  Re-positioned keys are compared with the oracle's
fp64 rotation of the same slab: the kernel rotates in fp32 (fp64 angles) and
rounds once to the cache dtype, so each element is within half a unit in the last
place of the dtype plus fp32 rounding of the rotation (stated per test)."""

import math

import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2607_21848_gb300 import api
from tests import _gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_21848_gb300 import build
    build.build()


def _segments(Nc, k):
    return [(0, Nc, api.SEG_SINK, 0)] + [((1 + r) * Nc, Nc, api.SEG_RETRIEVED, r) for r in range(k)] + \
           [((1 + k) * Nc, 2 * Nc, api.SEG_WINDOW, 0)]


def _setup(dtype, L=2, H=3, d=64, F=2, h=4, w=9, k=3, P=5, seed=3):
    Nc = F * h * w
    segs = _segments(Nc, k)
    Nk = (3 + k) * Nc
    cache = api.Cache.empty(L, Nk, H, d, dtype, segs)
    cache.k.fill_(-3.0)
    cache.v.fill_(-5.0)
    g = torch.Generator().manual_seed(seed)
    pool = torch.randn(P, 2, L, Nc, H, d, generator=g).to(dtype).cuda()
    shp = api.shape(L, H, d, F, h, w, dtype)
    return cache, pool, shp, Nc


def _rope_dict(rope, F):
    return dict(channel0=rope.channel0, pairs=rope.pairs, theta=rope.theta, interleaved=bool(rope.interleaved),
                pos_slot0=rope.pos_slot0, pos_stride=rope.pos_stride, frame_pos0=rope.frame_pos0, F=F)


def _check_keys(got, want, dtype, scale):
    """got: device keys in the cache dtype; want: the oracle's fp64 keys."""
    g = got.double().cpu().numpy()
    if dtype == torch.bfloat16:
        # half a bf16 ulp (<= 2^-8 relative) plus fp32 rotation error
        np.testing.assert_allclose(g, want, rtol=2.0 ** -8, atol=1e-6 * scale)
        exact = (got.cpu() == torch.from_numpy(want).to(torch.bfloat16)).float().mean().item()
        assert exact > 0.99, f"only {exact:.4f} of the keys equal the rounded oracle"
    else:
        np.testing.assert_allclose(g, want, rtol=1e-6, atol=1e-6 * scale)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_mirror_gather_is_byte_exact_and_skips_empty_slots(dtype):
    cache, pool, shp, Nc = _setup(dtype)
    idx = torch.tensor([7, -1, 2], dtype=torch.int32, device="cuda")
    api.crc_gather(shp, pool, idx, 3, cache)
    torch.cuda.synchronize()
    ref = oracle.gather(pool.cpu().double().numpy(), np.array([7, -1, 2]), pool.shape[0])
    for r in (0, 2):
        seg = slice((1 + r) * Nc, (2 + r) * Nc)
        assert torch.equal(cache.k[:, seg].cpu(), torch.from_numpy(ref[r][0]).to(dtype))
        assert torch.equal(cache.v[:, seg].cpu(), torch.from_numpy(ref[r][1]).to(dtype))
    # the empty slot, the sink and the window keep their contents
    assert bool((cache.k[:, 2 * Nc:3 * Nc] == -3.0).all()) and bool((cache.v[:, 2 * Nc:3 * Nc] == -5.0).all())
    assert bool((cache.k[:, :Nc] == -3.0).all()) and bool((cache.v[:, 4 * Nc:] == -5.0).all())


def _ropes(dtype, d):
    epv = 8 if dtype == torch.bfloat16 else 4
    return [
        # interleaved pairs from channel 0 (the temporal block of a 3-axis rotary layout)
        api.rope_params(0, d // 6 + 1, 10000.0, True, pos_slot0=40, pos_stride=2, frame_pos0=0),
        # interleaved block that starts mid-vector and ends mid-vector
        api.rope_params(2, 9, 500.0, True, pos_slot0=-5, pos_stride=3, frame_pos0=7),
        # half-split pairs (c, c + pairs), aligned to the 16-byte vectors
        api.rope_params(epv, 2 * epv, 10000.0, False, pos_slot0=100, pos_stride=2, frame_pos0=-4),
    ]


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_rope_repositioning_matches_oracle(dtype):
    d = 64
    for rope in _ropes(dtype, d):
        cache, pool, shp, Nc = _setup(dtype, d=d)
        chunks = [11, 3, -1]
        idx = torch.tensor(chunks, dtype=torch.int32, device="cuda")
        api.crc_gather(shp, pool, idx, 3, cache, rope=rope)
        torch.cuda.synchronize()
        pool64 = pool.cpu().double().numpy()
        ref = oracle.gather(pool64, np.array(chunks), pool.shape[0], rope=_rope_dict(rope, 2))
        scale = float(np.abs(pool64).max())
        for r in (0, 1):
            seg = slice((1 + r) * Nc, (2 + r) * Nc)
            _check_keys(cache.k[:, seg], ref[r][0], dtype, scale)
            # values carry no rotary embedding: byte-exact
            assert torch.equal(cache.v[:, seg].cpu(), torch.from_numpy(ref[r][1]).to(dtype))
            # channels outside the temporal block are copied bit for bit
            c0, np_ = rope.channel0, rope.pairs
            outside = list(range(0, c0)) + list(range(c0 + 2 * np_, d))
            src = pool[chunks[r] % pool.shape[0], 0]
            assert torch.equal(cache.k[:, seg][..., outside].cpu(), src[..., outside].cpu())
        assert bool((cache.k[:, 3 * Nc:4 * Nc] == -3.0).all())


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_unrotated_pairs_keep_their_bits_next_to_rotated_ones(dtype):
    """A temporal block that starts and ends inside 16-byte vectors (channels 2-19): the
    pairs it does not cover in those vectors (channels 0-1 and 20-23) must keep their bits,
    even for -0, infinities, NaN and subnormals, which a rotation by angle 0 would not."""
    d = 64
    cache, pool, shp, Nc = _setup(dtype, d=d)
    specials = torch.tensor([-0.0, float("inf"), float("-inf"), float("nan"), -1e-40, 0.0, -3.5, 1e30])
    k = pool[:, 0]
    for n, ch in enumerate([0, 1, 20, 21, 22, 23]):
        k[..., ch] = specials.roll(n)[torch.arange(k[..., ch].numel()) % len(specials)].reshape(k[..., ch].shape).to(dtype).cuda()
    rope = api.rope_params(2, 9, 500.0, True, pos_slot0=-5, pos_stride=3, frame_pos0=7)
    chunks = [11, 3, -1]
    api.crc_gather(shp, pool, torch.tensor(chunks, dtype=torch.int32, device="cuda"), 3, cache, rope=rope)
    torch.cuda.synchronize()
    ibits = torch.int16 if dtype == torch.bfloat16 else torch.int32
    for r in (0, 1):
        seg = slice((1 + r) * Nc, (2 + r) * Nc)
        got = cache.k[:, seg].contiguous().view(ibits)
        src = pool[chunks[r] % pool.shape[0], 0].contiguous().view(ibits)
        outside = [0, 1] + list(range(20, d))
        assert torch.equal(got[..., outside], src[..., outside])
        # and the block itself was moved: its bits differ from the slab's
        assert not torch.equal(got[..., 2:20], src[..., 2:20])


def test_zero_shift_is_a_plain_copy():
    # slot 0 holding chunk 5 at pos_slot0 = frame_pos0 + 5 F is not moved: byte-exact
    dtype = torch.bfloat16
    cache, pool, shp, Nc = _setup(dtype)
    rope = api.rope_params(0, 16, 10000.0, True, pos_slot0=10 + 5 * 2, pos_stride=2, frame_pos0=10)
    api.crc_gather(shp, pool, torch.tensor([5, 6, -1], dtype=torch.int32, device="cuda"), 3, cache, rope=rope)
    torch.cuda.synchronize()
    assert torch.equal(cache.k[:, Nc:2 * Nc], pool[0, 0])
    # slot 1 holds chunk 6: shift (20 + 1 * 2) - (10 + 6 * 2) = 0 as well
    assert torch.equal(cache.k[:, 2 * Nc:3 * Nc], pool[1, 0])


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_retrieve_and_mirror_gather_agree_bitwise(dtype):
    wl = synth.make_workload(2, bank=12)
    cache, _, shp, Nc = _setup(dtype)
    mirror = api.Cache.empty(cache.k.shape[0], cache.n_keys, cache.k.shape[2], cache.k.shape[3], dtype,
                             cache.segments)
    bank = api.Bank(16, 2, 4, 9, shp.L, shp.H, shp.d, dtype, 5)
    bank.kv.copy_(torch.randn(bank.kv.shape, generator=torch.Generator().manual_seed(9)).to(dtype))
    fr = synth.Frames(wl.bank_frames.K[:, :2], wl.bank_frames.R[:, :2], wl.bank_frames.c[:, :2])
    _gpu.insert_poses(bank, shp, fr)
    rope = api.rope_params(0, 11, 10000.0, True, pos_slot0=30, pos_stride=2)
    params = api.retrieval_params(1.0, 0.5, math.inf, -1.0, 1, 3, 6, 2)
    idx = torch.zeros(3, dtype=torch.int32, device="cuda")
    count = torch.zeros(1, dtype=torch.int32, device="cuda")
    api.crc_retrieve(bank, 12, shp, synth.frame_records(fr[7]), 12, params, cache, idx, None, count, rope=rope)
    api.crc_gather(shp, bank.kv, idx, 3, mirror, rope=rope)
    torch.cuda.synchronize()
    seg = slice(Nc, 4 * Nc)
    assert torch.equal(cache.k[:, seg], mirror.k[:, seg]) and torch.equal(cache.v[:, seg], mirror.v[:, seg])
    # and the fused gather matches the oracle's re-positioning of the retrieved chunks
    slots = idx.cpu().numpy()
    ref = oracle.gather(bank.kv.cpu().double().numpy(), slots, 5, rope=_rope_dict(rope, 2))
    for r in range(3):
        _check_keys(cache.k[:, (1 + r) * Nc:(2 + r) * Nc], ref[r][0], dtype, float(bank.kv.abs().max()))


def test_mirror_of_a_control_cache_with_fewer_layers():
    # the mirrored cache has its own layer count (e.g. only the control blocks)
    dtype = torch.bfloat16
    cache, pool, shp, Nc = _setup(dtype, L=5)
    ctl, ctl_pool, ctl_shp, _ = _setup(dtype, L=2, seed=4)
    idx = torch.tensor([4, 8, 1], dtype=torch.int32, device="cuda")
    api.crc_gather(shp, pool, idx, 3, cache)
    api.crc_gather(ctl_shp, ctl_pool, idx, 3, ctl)
    torch.cuda.synchronize()
    for r, j in enumerate([4, 8, 1]):
        seg = slice((1 + r) * Nc, (2 + r) * Nc)
        assert torch.equal(cache.k[:, seg], pool[j % 5, 0]) and torch.equal(ctl.k[:, seg], ctl_pool[j % 5, 0])
        assert torch.equal(ctl.v[:, seg], ctl_pool[j % 5, 1])


def test_full_size_wan13b_repositioned_gather_sampled():
    # Wan-1.3B chunk shape, all 30 layers, 22 interleaved temporal pairs; sampled rows vs the oracle
    wl = synth.make_workload(2, layers=30)
    dtype = torch.bfloat16
    Nc, L, H, d = wl.Nc, wl.L, wl.H, wl.d
    segs = _segments(Nc, 1)
    cache = api.Cache.empty(L, 4 * Nc, H, d, dtype, segs)
    g = torch.Generator(device="cuda").manual_seed(5)
    pool = (torch.randn(4, 2, L, Nc, H, d, generator=g, device="cuda") * wl.qkv_scale).to(dtype)
    shp = api.shape(L, H, d, wl.F, wl.h, wl.w, dtype)
    rope = api.rope_params(0, 22, 10000.0, True, pos_slot0=3 * 64 - 3, pos_stride=3)
    api.crc_gather(shp, pool, torch.tensor([33], dtype=torch.int32, device="cuda"), 1, cache, rope=rope)
    torch.cuda.synchronize()
    rows = np.random.default_rng(0).choice(Nc, 64, replace=False)
    rows_t = torch.from_numpy(rows).cuda()
    for layer in (0, 17, 29):
        src = pool[33 % 4, :, layer, rows_t].cpu().double().numpy()[:, None]  # [2, 1, rows, H, d]
        ref = oracle.gather(src[None], np.array([33]), 1, rope=_rope_dict(rope, wl.F))[0]
        # the oracle's positions depend on the chunk and slot only, not on the row subset
        _check_keys(cache.k[layer, Nc + rows_t], ref[0][0], dtype, float(np.abs(src).max()))
        assert torch.equal(cache.v[layer, Nc + rows_t].cpu(),
                           torch.from_numpy(ref[1][0]).to(dtype))


@pytest.mark.parametrize("bad, status", [
    (dict(channel0=1, pairs=4, interleaved=True), api.CrcError),   # odd start of interleaved pairs
    (dict(channel0=0, pairs=40, interleaved=True), api.CrcError),  # 80 channels > d = 64
    (dict(channel0=4, pairs=8, interleaved=False), api.CrcError),  # half-split not on a 16-byte vector
    (dict(channel0=0, pairs=65, interleaved=True), api.CrcError),  # above CRC_MAX_ROPE_PAIRS
])
def test_bad_rope_layouts_are_rejected_before_launch(bad, status):
    dtype = torch.bfloat16
    cache, pool, shp, Nc = _setup(dtype)
    rope = api.rope_params(bad["channel0"], bad["pairs"], 10000.0, bad["interleaved"], 0, 1)
    before = cache.k.clone()
    with pytest.raises(status):
        api.crc_gather(shp, pool, torch.zeros(3, dtype=torch.int32, device="cuda"), 3, cache, rope=rope)
    torch.cuda.synchronize()
    assert torch.equal(before, cache.k)


def test_gather_rejects_bad_slot_count():
    cache, pool, shp, Nc = _setup(torch.float32)
    for k in (0, 9):
        with pytest.raises(api.CrcError):
            api.crc_gather(shp, pool, torch.zeros(9, dtype=torch.int32, device="cuda"), k, cache)


def test_exclude_sink_matches_oracle():
    wl = synth.make_workload(2, bank=12)
    bank, shp = _gpu.make_bank(wl, torch.bfloat16)
    # every chunk at the current pose: chunk 0 wins the tie unless excluded
    cur = wl.bank_frames[5]
    fr = synth.Frames(np.repeat(cur.K[None], 12, 0), np.repeat(cur.R[None], 12, 0), np.repeat(cur.c[None], 12, 0))
    _gpu.insert_poses(bank, shp, fr)
    bc, bv = _gpu.oracle_bank_poses(fr)
    cn, vn = oracle.chunk_pose(cur.R, cur.c)
    for excl in (False, True):
        oi, _, oc = oracle.retrieve(bc, bv, cn, vn, 12, 1.0, 0.5, math.inf, -1.0, 1, 2, exclude_sink=excl)
        params = api.retrieval_params(1.0, 0.5, math.inf, -1.0, 1, 2, exclude_sink=excl)
        idx = torch.zeros(2, dtype=torch.int32, device="cuda")
        count = torch.zeros(1, dtype=torch.int32, device="cuda")
        api.crc_retrieve(bank, 12, shp, synth.frame_records(cur), 12, params, None, idx, None, count)
        torch.cuda.synchronize()
        assert int(count.item()) == oc and list(idx.cpu().numpy()) == list(oi)
        assert (0 in list(oi)) != excl
