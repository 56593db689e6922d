"""GPU parity of the bank, the retrieval (Eq. 1) and the gather against the oracle:
bit-exact pose summaries, indices, counts and scores; byte-exact gathers."""

import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2607_21848_gb300 import _abi, api
from tests import _gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_21848_gb300 import build
    build.build()


def _read_poses(bank, B):
    return bank.centre[:B].cpu().numpy(), bank.view[:B].cpu().numpy()


@pytest.mark.parametrize("cfg", [1, 2, 3, 4, 5])
def test_pose_summary_bit_exact(cfg):
    wl = synth.make_workload(cfg)
    bank, shp = _gpu.make_bank(wl, _gpu.dev_dtype(wl))
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    torch.cuda.synchronize()
    c, v = _read_poses(bank, wl.bank_size)
    oc, ov = _gpu.oracle_bank_poses(wl.bank_frames)
    np.testing.assert_array_equal(c, oc)
    np.testing.assert_array_equal(v, ov)
    rec = bank.frames.cpu().numpy().reshape(-1, 21)
    np.testing.assert_array_equal(rec, synth.frame_records(wl.bank_frames))


def _gpu_retrieve(wl, bank, shp, bank_count, n, cur, k, ext_first=-1, ext_min=0, cache=None, **over):
    p = dict(E=wl.E, w_v=wl.w_v, tau_c=wl.tau_c, cos_tau_v=wl.cos_tau_v, delta=wl.delta)
    p.update(over)
    params = api.retrieval_params(p["E"], p["w_v"], p["tau_c"], p["cos_tau_v"], p["delta"], k, ext_first, ext_min)
    idx = torch.full((k,), -7, dtype=torch.int32, device="cuda")
    score = torch.zeros(k, dtype=torch.float64, device="cuda")
    count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    api.crc_retrieve(bank, bank_count, shp, synth.frame_records(cur), n, params, cache, idx, score, count)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), score.cpu().numpy(), int(count.item())


@pytest.mark.parametrize("cfg", [1, 2, 3, 4])
def test_retrieve_topk_bit_exact(cfg):
    wl = synth.make_workload(cfg)
    bank, shp = _gpu.make_bank(wl, _gpu.dev_dtype(wl))
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    for k in sorted({wl.k, 1, 5, _abi.CRC_MAX_K}):
        oi, os_, oc, _ = _gpu.oracle_retrieve(wl, k=k)
        gi, gs, gc = _gpu_retrieve(wl, bank, shp, wl.bank_size, wl.n, wl.cur_frames, k)
        assert gc == oc
        np.testing.assert_array_equal(gi, oi)
        np.testing.assert_array_equal(gs, os_)  # bit-exact fp64 scores


@pytest.mark.parametrize("over", [dict(tau_c=2.0), dict(cos_tau_v=math.cos(math.radians(20))), dict(delta=40),
                                  dict(tau_c=0.0), dict(E=7.5, w_v=0.0), dict(E=0.3, w_v=3.0)])
def test_retrieve_gates_bit_exact(over):
    wl = synth.make_workload(3)
    bank, shp = _gpu.make_bank(wl, torch.bfloat16)
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    oi, os_, oc, _ = _gpu.oracle_retrieve(wl, k=4, **over)
    gi, gs, gc = _gpu_retrieve(wl, bank, shp, wl.bank_size, wl.n, wl.cur_frames, 4, **over)
    assert gc == oc
    np.testing.assert_array_equal(gi, oi)
    np.testing.assert_array_equal(gs, os_)


def _random_bank(B, seed, ties=0):
    """B entries with random centres and unit view directions; with `ties`, runs of
    entries share one pose (identical scores) spread over the whole bank."""
    g = np.random.default_rng(seed)
    c = g.normal(size=(B, 3)) * 20.0
    v = g.normal(size=(B, 3))
    v /= np.linalg.norm(v, axis=1, keepdims=True)
    pos = np.zeros(3)
    if ties:  # the tied entries share the pose of a camera at c[pick[0]] looking along +x
        pick = g.choice(B, ties, replace=False)
        pos = c[pick[0]].copy()
        c[pick] = pos
        v[pick] = [1.0, 0.0, 0.0]
    return c, v, pos


@pytest.mark.parametrize("B,k,ties", [(513, 3, 0), (4097, 8, 0), (100003, 3, 0), (100003, 8, 0), (20000, 8, 40)])
def test_retrieve_large_banks_bit_exact(B, k, ties):
    """Banks of more than 512 entries are scored by many blocks whose candidates meet in the
    workspace: indices, count and fp64 scores bit-exact against the oracle, ties across
    blocks broken by the chunk index, and every gate in force."""
    c, v, pos = _random_bank(B, seed=B + k, ties=ties)
    bank = api.Bank(B, 3, 8, 8, 1, 1, 64, torch.float32, 1, with_kv=False)
    bank.centre.copy_(torch.from_numpy(c))
    bank.view.copy_(torch.from_numpy(v))
    assert bank.workspace is not None
    shp = api.shape(1, 1, 64, 3, 8, 8, torch.float32)
    K = synth.pinhole(8, 8, 90.0)
    # the current chunk looks along +x from the tied pose (or the origin)
    cur = synth.Frames(np.stack([K] * 3), np.stack([synth.camera_rotation(0.0)] * 3), np.stack([pos] * 3))
    cn, vn = oracle.chunk_pose(cur.R, cur.c)
    for over in (dict(E=10.0, w_v=0.5, tau_c=math.inf, cos_tau_v=-1.0, delta=1),
                 dict(E=10.0, w_v=0.5, tau_c=3.0, cos_tau_v=math.cos(math.radians(60)), delta=B // 3)):
        n = B + 5
        oi, os_, oc = oracle.retrieve(c, v, cn, vn, n, k=k, **over)
        params = api.retrieval_params(over["E"], over["w_v"], over["tau_c"], over["cos_tau_v"], over["delta"], k)
        idx = torch.full((k,), -7, dtype=torch.int32, device="cuda")
        score = torch.zeros(k, dtype=torch.float64, device="cuda")
        count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
        api.crc_retrieve(bank, B, shp, synth.frame_records(cur), n, params, None, idx, score, count)
        torch.cuda.synchronize()
        assert int(count.item()) == oc
        np.testing.assert_array_equal(idx.cpu().numpy(), oi)
        np.testing.assert_array_equal(score.cpu().numpy(), os_)
        if ties and math.isinf(over["tau_c"]):
            assert oc == k and len(set(os_[:k])) == 1  # k equal scores (0), ordered by j


def test_retrieve_admits_only_chunks_whose_slab_still_holds_them():
    """A bank of 12 chunks with a pool of 4 tracked K/V slabs: after 12 updates only the
    last 4 chunks are held.  Retrieval admits only those (the oracle over the resident
    chunks), the window-extension fallback skips chunks that are no longer held, and the
    gathered K/V are each chunk's own."""
    F, h, w, L, H, d, P, B = 3, 8, 8, 1, 2, 64, 4, 12
    Nc = F * h * w
    K = synth.pinhole(h, w, 90.0)
    fr = synth.random_walk(synth.rng(77, "poses"), B, F, K, step=0.3, radius=3.0)
    shp = api.shape(L, H, d, F, h, w, torch.float32)
    bank = api.Bank(B, F, h, w, L, H, d, torch.float32, P, track_slabs=True)
    g = torch.Generator(device="cuda").manual_seed(9)
    kv = [(torch.randn(L, Nc, H, d, generator=g, device="cuda"), torch.randn(L, Nc, H, d, generator=g, device="cuda"))
          for _ in range(B)]
    depth = torch.ones(F, h, w, device="cuda")
    for j in range(B):
        api.crc_cache_update(bank, shp, j, synth.frame_records(fr[j]), depth, kv[j][0], kv[j][1], None, -1)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bank.slab_chunk.cpu().numpy(), [8, 9, 10, 11])
    resident = np.zeros(B, bool)
    resident[B - P:] = True
    bc, bv = _gpu.oracle_bank_poses(fr)
    cur = fr[3]
    cn, vn = oracle.chunk_pose(cur.R, cur.c)
    k = 3
    segs = [(0, Nc, api.SEG_SINK, 0)] + [((1 + r) * Nc, Nc, api.SEG_RETRIEVED, r) for r in range(k)]
    for n, delta, ext_first in ((B, 1, -1), (B, 5, 9), (B, 3, 10)):  # [8..11] top-3; [9, 8, -]; [8, 9] + 10
        oi, os_, oc = oracle.retrieve(bc, bv, cn, vn, n, 1.0, 0.5, math.inf, -1.0, delta, k, resident=resident)
        slots = oracle.fill_slots(oi, oc, ext_first, 1, resident=resident)
        cache = api.Cache.empty(L, (1 + k) * Nc, H, d, torch.float32, segs)
        params = api.retrieval_params(1.0, 0.5, math.inf, -1.0, delta, k, ext_first, 1)
        idx = torch.full((k,), -7, dtype=torch.int32, device="cuda")
        count = torch.zeros(1, dtype=torch.int32, device="cuda")
        api.crc_retrieve(bank, B, shp, synth.frame_records(cur), n, params, cache, idx, None, count)
        torch.cuda.synchronize()
        gi = idx.cpu().numpy()
        assert int(count.item()) == oc
        np.testing.assert_array_equal(gi, slots)
        assert all(resident[j] for j in gi if j >= 0)
        for r, j in enumerate(gi):
            if j >= 0:
                off = (1 + r) * Nc
                assert torch.equal(cache.k[:, off:off + Nc], kv[j][0])
                assert torch.equal(cache.v[:, off:off + Nc], kv[j][1])
    # without the owner array every chunk is admissible (the caller vouches for the slabs)
    untracked = api.Bank(B, F, h, w, L, H, d, torch.float32, P)
    untracked.centre.copy_(bank.centre)
    untracked.view.copy_(bank.view)
    oi, _, oc = oracle.retrieve(bc, bv, cn, vn, B, 1.0, 0.5, math.inf, -1.0, 1, k)
    idx = torch.full((k,), -7, dtype=torch.int32, device="cuda")
    count = torch.zeros(1, dtype=torch.int32, device="cuda")
    api.crc_retrieve(untracked, B, shp, synth.frame_records(cur), B,
                     api.retrieval_params(1.0, 0.5, math.inf, -1.0, 1, k), None, idx, None, count)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    assert not all(resident[j] for j in oi)  # the sub-bank and the whole bank differ here


def test_retrieve_stream_gates_and_window_extension():
    wl = synth.make_workload(5)
    bank, shp = _gpu.make_bank(wl, torch.bfloat16)
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    seen_full = seen_empty = False
    for n in list(range(0, 12)) + [60, 148, 150, 151, 152, 155, 170, 199]:
        ext = n - 2 if n - 2 >= 1 else -1
        oi, os_, oc, slots = _gpu.oracle_retrieve(wl, bank_count=n + 1, n=n, k=wl.k, ext_first=ext, ext_min=1)
        gi, gs, gc = _gpu_retrieve(wl, bank, shp, n + 1, n, wl.bank_frames[n], wl.k, ext_first=ext, ext_min=1)
        assert gc == oc, n
        np.testing.assert_array_equal(gi, slots)
        np.testing.assert_array_equal(gs[:oc], os_[:oc])
        assert np.all(np.isinf(gs[oc:]))
        seen_full |= oc == wl.k
        seen_empty |= oc == 0
    assert seen_full and seen_empty  # the loop closes after one lap; before that A_n is empty


def test_retrieve_handworked_golden():
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "retrieval_handworked.json")))
    K = synth.pinhole(8, 8, 90.0)
    bank_fr = synth.Frames(np.stack([K] * 3)[:, None], np.stack(
        [synth.camera_rotation(math.radians(e["yaw_deg"])) for e in g["bank"]])[:, None],
        np.array([e["c"] for e in g["bank"]])[:, None])
    cur = synth.Frames(K[None], synth.camera_rotation(0.0)[None], np.array([g["current"]["c"]]))
    bank = api.Bank(4, 1, 8, 8, 1, 1, 64, torch.float32, 1, with_kv=False)
    shp = api.shape(1, 1, 64, 1, 8, 8, torch.float32)
    api.crc_bank_insert_poses(bank, shp, 0, synth.frame_records(bank_fr))
    for case in g["cases"]:
        k = case["k"]
        tau = math.inf if case["tau_c"] == "inf" else case["tau_c"]
        params = api.retrieval_params(case["E"], g["w_v"], tau, case["cos_tau_v"], case["delta"], k)
        idx = torch.zeros(k, dtype=torch.int32, device="cuda")
        score = torch.zeros(k, dtype=torch.float64, device="cuda")
        count = torch.zeros(1, dtype=torch.int32, device="cuda")
        api.crc_retrieve(bank, 3, shp, synth.frame_records(cur), g["n"], params, None, idx, score, count)
        torch.cuda.synchronize()
        assert count.item() == case["count"]
        assert list(idx.cpu().numpy()) == case["idx"]
        exp = np.array([math.inf if s == "inf" else s for s in case["score"]])
        np.testing.assert_allclose(score.cpu().numpy()[np.isfinite(exp)], exp[np.isfinite(exp)], atol=1e-12)


def test_retrieve_empty_bank_and_ties():
    wl = synth.make_workload(2)
    bank, shp = _gpu.make_bank(wl, torch.bfloat16)
    gi, gs, gc = _gpu_retrieve(wl, bank, shp, 0, wl.n, wl.cur_frames, 2, ext_first=5, ext_min=3)
    assert gc == 0 and list(gi) == [5, 4]
    # identical poses: ties break toward the smaller chunk index
    fr = synth.Frames(np.repeat(wl.bank_frames.K[:1], 6, 0), np.repeat(wl.bank_frames.R[:1], 6, 0),
                      np.repeat(wl.bank_frames.c[:1], 6, 0))
    _gpu.insert_poses(bank, shp, fr)
    gi, gs, gc = _gpu_retrieve(wl, bank, shp, 6, 10, wl.bank_frames[0], 4)
    assert gc == 4 and list(gi) == [0, 1, 2, 3]
    assert np.all(gs == gs[0])


def _gather_setup(dtype, L=2, H=3, d=64, F=2, h=4, w=8, k=3, P=5):
    Nc = F * h * w
    segs = [(0, Nc, api.SEG_SINK, 0)] + [((1 + r) * Nc, Nc, api.SEG_RETRIEVED, r) for r in range(k)] + \
           [((1 + k) * Nc, Nc, api.SEG_WINDOW, 0)]
    Nk = (2 + k) * Nc
    cache = api.Cache.empty(L, Nk, H, d, dtype, segs)
    cache.k.fill_(-3.0)
    cache.v.fill_(-5.0)
    bank = api.Bank(16, F, h, w, L, H, d, dtype, P)
    bank.kv.copy_(torch.randn(bank.kv.shape, generator=torch.Generator().manual_seed(3)).to(dtype))
    shp = api.shape(L, H, d, F, h, w, dtype)
    return cache, bank, shp, segs, Nc


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_gather_copies_slabs_and_fills_window_extension(dtype):
    wl = synth.make_workload(2, bank=12)
    cache, bank, shp, segs, Nc = _gather_setup(dtype)
    fr = synth.Frames(wl.bank_frames.K[:, :2], wl.bank_frames.R[:, :2], wl.bank_frames.c[:, :2])
    _gpu.insert_poses(bank, shp, fr)
    cur = fr[7]
    # tight distance gate: only a few admissible chunks, the rest of the slots extend the window
    bc, bv = _gpu.oracle_bank_poses(fr)
    cn, vn = oracle.chunk_pose(cur.R, cur.c)
    for tau in (math.inf, 0.6, 0.0):
        oi, _, oc = oracle.retrieve(bc, bv, cn, vn, 12, 1.0, 0.5, tau, -1.0, 1, 3)
        slots = oracle.fill_slots(oi, oc, 6, 2)
        params = api.retrieval_params(1.0, 0.5, tau, -1.0, 1, 3, 6, 2)
        idx = torch.zeros(3, dtype=torch.int32, device="cuda")
        count = torch.zeros(1, dtype=torch.int32, device="cuda")
        api.crc_retrieve(bank, 12, shp, synth.frame_records(cur), 12, params, cache, idx, None, count)
        torch.cuda.synchronize()
        assert count.item() == oc and list(idx.cpu().numpy()) == list(slots)
        pool = bank.kv.cpu()
        ref = oracle.gather(pool.float().numpy(), slots, bank.num_slabs)
        for r in range(3):
            seg = cache.k[:, (1 + r) * Nc:(2 + r) * Nc].cpu()
            segv = cache.v[:, (1 + r) * Nc:(2 + r) * Nc].cpu()
            assert torch.equal(seg, torch.from_numpy(ref[r][0]).to(dtype))
            assert torch.equal(segv, torch.from_numpy(ref[r][1]).to(dtype))
        # sink and window untouched
        assert bool((cache.k[:, :Nc] == -3.0).all()) and bool((cache.v[:, 4 * Nc:] == -5.0).all())


def test_cache_update_writes_window_slab_depth_and_poses():
    wl = synth.make_workload(2, bank=12)
    dtype = torch.bfloat16
    cache, bank, shp, segs, Nc = _gather_setup(dtype, k=1)
    fr = synth.Frames(wl.bank_frames.K[:, :2], wl.bank_frames.R[:, :2], wl.bank_frames.c[:, :2])
    g = torch.Generator().manual_seed(9)
    knew = torch.randn(2, Nc, 3, 64, generator=g).to(dtype).cuda()
    vnew = torch.randn(2, Nc, 3, 64, generator=g).to(dtype).cuda()
    depth = torch.rand(2, 4, 8, generator=g).cuda() * 10
    before = bank.kv.clone()
    api.crc_cache_update(bank, shp, 7, synth.frame_records(fr[7]), depth, knew, vnew, cache, 2 * Nc)
    torch.cuda.synchronize()
    assert torch.equal(cache.k[:, 2 * Nc:3 * Nc], knew) and torch.equal(cache.v[:, 2 * Nc:3 * Nc], vnew)
    assert bool((cache.k[:, :2 * Nc] == -3.0).all())  # sink and retrieved slot untouched
    slab = 7 % bank.num_slabs
    assert torch.equal(bank.kv[slab, 0], knew) and torch.equal(bank.kv[slab, 1], vnew)
    others = [i for i in range(bank.num_slabs) if i != slab]
    assert torch.equal(bank.kv[others], before[others])
    assert torch.equal(bank.depth[7], depth)
    oc, ov = oracle.chunk_pose(fr[7].R, fr[7].c)
    np.testing.assert_array_equal(bank.centre[7].cpu().numpy(), oc)
    np.testing.assert_array_equal(bank.view[7].cpu().numpy(), ov)
    # poses-only update leaves the cache alone
    api.crc_cache_update(bank, shp, 8, synth.frame_records(fr[8]), depth, None, None, None, -1)
    torch.cuda.synchronize()
    oc, ov = oracle.chunk_pose(fr[8].R, fr[8].c)
    np.testing.assert_array_equal(bank.centre[8].cpu().numpy(), oc)


def test_host_validation_rejects_bad_arguments():
    wl = synth.make_workload(2, bank=4)
    bank, shp = _gpu.make_bank(wl, torch.bfloat16)
    params = api.retrieval_params(1.0, 0.5, math.inf, -1.0, 1, 0)  # k = 0
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    count = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(api.CrcError):
        api.crc_retrieve(bank, 4, shp, synth.frame_records(wl.cur_frames), 4, params, None, idx, None, count)
    params = api.retrieval_params(0.0, 0.5, math.inf, -1.0, 1, 1)  # E = 0
    with pytest.raises(api.CrcError):
        api.crc_retrieve(bank, 4, shp, synth.frame_records(wl.cur_frames), 4, params, None, idx, None, count)
    params = api.retrieval_params(1.0, 0.5, math.inf, -1.0, 1, 1)
    with pytest.raises(api.CrcError):  # bank_count beyond capacity
        api.crc_retrieve(bank, 5, shp, synth.frame_records(wl.cur_frames), 4, params, None, idx, None, count)
    bad = synth.frame_records(wl.cur_frames).copy()
    bad[0, 18] = np.nan
    with pytest.raises(api.CrcError):
        api.crc_retrieve(bank, 4, shp, bad, 4, params, None, idx, None, count)
