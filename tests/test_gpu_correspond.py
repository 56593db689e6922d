"""GPU parity of the reprojection correspondence (Eq. 3-4) against the oracle.

Landing cells and valid flags must be identical except for pairs whose integer
decision lies within rounding distance of a boundary (u^ + 1/2 within 1e-4 of an
integer, or the depth / visibility comparison within 1e-6 / 1e-5 relative);
u^ of pairs valid on both sides must agree to 1e-3 token."""

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


def _run(wl, slots, count, eps, cur=None, depth_cur=None, fill_depth=True):
    dtype = _gpu.dev_dtype(wl)
    bank, shp = _gpu.make_bank(wl, dtype)
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    if fill_depth:
        for j in set(int(x) for x in slots if x >= 0):
            bank.depth[j] = torch.from_numpy(wl.depth_of(j)).cuda()
    cur = wl.cur_frames if cur is None else cur
    depth_cur = wl.depth_of(wl.n) if depth_cur is None else depth_cur
    k = len(slots)
    S = k * wl.F
    idx = torch.tensor(np.asarray(slots, dtype=np.int32), device="cuda")
    cnt = torch.tensor([count], dtype=torch.int32, device="cuda")
    uv = torch.full((wl.Nq, S, 2), -9.0, device="cuda")
    cell = torch.full((wl.Nq, S), -9, dtype=torch.int32, device="cuda")
    valid = torch.full((wl.Nq, S), 9, dtype=torch.uint8, device="cuda")
    api.crc_correspond(shp, synth.frame_records(cur), torch.from_numpy(depth_cur).cuda(), bank, idx, cnt, k, eps,
                       uv, cell, valid)
    torch.cuda.synchronize()
    return uv.cpu().numpy().astype(np.float64), cell.cpu().numpy(), valid.cpu().numpy()


@pytest.mark.parametrize("cfg", [1, 2, 3, 4, 5])
@pytest.mark.parametrize("eps_mode", ["config", "0.05"])
def test_correspond_matches_oracle(cfg, eps_mode):
    wl = synth.make_workload(cfg)
    eps = wl.eps if eps_mode == "config" else 0.05
    if cfg == 5:
        n = 160  # after the loop closes: two retrieved chunks
        _, _, count, slots = _gpu.oracle_retrieve(wl, bank_count=n + 1, n=n, ext_first=n - 2, ext_min=1)
        cur = wl.bank_frames[n]
        dcur = wl.depth_of(n)
    else:
        _, _, count, slots = _gpu.oracle_retrieve(wl)
        cur, dcur = wl.cur_frames, wl.depth_of(wl.n)
    assert count >= 1
    o = _gpu.oracle_correspond(wl, slots, count, eps=eps, cur=cur, depth_cur=dcur)
    g_uv, g_cell, g_valid = _run(wl, slots, count, eps, cur=cur, depth_cur=dcur)
    r = _gpu.compare_correspondence(wl, o, g_uv, g_cell, g_valid, eps, depth_cur=dcur)
    assert r["bad_valid"] == 0 and r["bad_cell"] == 0, r
    assert r["uv_err"] <= 1e-3, r
    assert r["n_valid"] > 0.05 * r["n"], r  # the workload exercises real correspondences
    assert r["exempt"] <= 0.01 * r["n"], r


def test_correspond_identity_pose_maps_token_to_itself():
    wl = synth.make_workload(2)
    j = 5
    fr = wl.bank_frames[j]
    dep = wl.depth_of(j)
    g_uv, g_cell, g_valid = _run(wl, [j], 1, 0.05, cur=fr, depth_cur=dep)
    ii, jj = np.meshgrid(np.arange(wl.h), np.arange(wl.w), indexing="ij")
    u = np.tile(np.stack([jj.ravel(), ii.ravel()], 1), (wl.F, 1))
    # same-frame pairs (t = s) map every token onto itself
    for t in range(wl.F):
        rows = slice(t * wl.h * wl.w, (t + 1) * wl.h * wl.w)
        np.testing.assert_allclose(g_uv[rows, t], u[rows], atol=2e-3)
        assert g_valid[rows, t].all()
        np.testing.assert_array_equal(g_cell[rows, t], np.arange(wl.h * wl.w))


def test_correspond_window_extension_and_empty_slots_are_invalid():
    wl = synth.make_workload(4)
    _, _, count, slots = _gpu.oracle_retrieve(wl)
    slots = np.array([slots[0], 3], dtype=np.int32)  # slot 1 holds a window-extension chunk
    g_uv, g_cell, g_valid = _run(wl, slots, 1, math.inf)
    assert g_valid[:, :wl.F].any() and not g_valid[:, wl.F:].any()
    assert (g_cell[:, wl.F:] == -1).all() and np.isnan(g_uv[:, wl.F:]).all()
    g_uv, g_cell, g_valid = _run(wl, np.array([-1, slots[0]], dtype=np.int32), 2, math.inf)
    assert not g_valid[:, :wl.F].any() and g_valid[:, wl.F:].any()


def test_correspond_bad_depth_is_invalid_not_undefined():
    wl = synth.make_workload(2)
    _, _, count, slots = _gpu.oracle_retrieve(wl)
    d = wl.depth_of(wl.n).copy()
    d[0, 0, :4] = [0.0, -2.0, np.nan, np.inf]
    g_uv, g_cell, g_valid = _run(wl, slots, count, 0.05, depth_cur=d)
    assert not g_valid[:4].any() and (g_cell[:4] == -1).all()


def _eight_chunk_scene(F=4, h=24, w=40, k=8, seed=999):
    """The reprojection sweep's structure at a smaller grid: k + 1 consecutive chunks of
    F frames along a ground random walk through the room scene, depth rendered from it."""
    from synth import workloads as W

    K = synth.pinhole(h, w, 90.0)
    fr = synth.random_walk(synth.rng(seed, "sweep"), k + 1, F, K, step=0.5, radius=24.0)
    scene = W.Scene.room(synth.rng(seed, "scene"), radius=40.0, n_walls=12, n_boards=60, board_rmin=2.0,
                         board_rmax=36.0)
    dep = np.stack([np.stack([W.render_depth(scene, fr.K[j, f], fr.R[j, f], fr.c[j, f], h, w, 0.5, 50.0)
                              for f in range(F)]) for j in range(k + 1)]).astype(np.float32)
    return fr, dep


@pytest.mark.parametrize("eps", [0.05, math.inf])
def test_correspond_four_frames_eight_slots_matches_oracle(eps):
    """F = 4 and k = 8 (S = 32: two frames per thread, four lane groups per query
    group) against the oracle, every pair."""
    import types

    F, h, w, k = 4, 24, 40, 8
    fr, dep = _eight_chunk_scene(F, h, w, k)
    bank = api.Bank(k + 1, F, h, w, 1, 1, 64, torch.float32, 1, device="cuda", with_kv=False)
    shp = api.shape(1, 1, 64, F, h, w, torch.float32)
    api.crc_bank_insert_poses(bank, shp, 0, synth.frame_records(fr))
    bank.depth.copy_(torch.from_numpy(dep).cuda())
    Nq, S = F * h * w, k * F
    idx = torch.arange(k, dtype=torch.int32, device="cuda")
    cnt = torch.tensor([k], dtype=torch.int32, device="cuda")
    uv = torch.full((Nq, S, 2), -9.0, device="cuda")
    cell = torch.full((Nq, S), -9, dtype=torch.int32, device="cuda")
    valid = torch.full((Nq, S), 9, dtype=torch.uint8, device="cuda")
    api.crc_correspond(shp, synth.frame_records(fr[k]), bank.depth[k].clone(), bank, idx, cnt, k, eps, uv, cell,
                       valid)
    torch.cuda.synchronize()
    cur = fr[k]
    Ks = fr.K[:k].reshape(S, 3, 3)
    Rs = fr.R[:k].reshape(S, 3, 3)
    cs = fr.c[:k].reshape(S, 3)
    ouv, ocell, ovalid, zs = oracle.correspond(dep[k], cur.K, cur.R, cur.c, dep[:k].reshape(S, h, w), Ks, Rs, cs,
                                               eps, with_zs=True)
    o = (ouv, ocell, ovalid, zs, dep[:k].reshape(S, h, w), np.ones(S, bool))
    geo = types.SimpleNamespace(w=w, h=h, n=k, depth_of=lambda j: dep[j])
    r = _gpu.compare_correspondence(geo, o, uv.cpu().numpy().astype(np.float64), cell.cpu().numpy(),
                                    valid.cpu().numpy(), eps, depth_cur=dep[k])
    assert r["bad_valid"] == 0 and r["bad_cell"] == 0, r
    assert r["uv_err"] <= 1e-3, r
    assert r["n_valid"] > 0.5 * r["n"] and r["exempt"] <= 0.01 * r["n"], r


def test_correspond_unaligned_outputs_and_no_cell_are_bit_identical():
    """Outputs that only allow narrower stores (u^ 8-byte aligned, cell 4-byte, flags
    1-byte) and a NULL cell array give the same bytes as the aligned call."""
    wl = synth.make_workload(4)  # S = 6: two source frames per thread when aligned
    _, _, count, slots = _gpu.oracle_retrieve(wl)
    ref = _run(wl, slots, count, 0.05)
    dtype = _gpu.dev_dtype(wl)
    bank, shp = _gpu.make_bank(wl, dtype)
    _gpu.insert_poses(bank, shp, wl.bank_frames)
    for j in set(int(x) for x in slots if x >= 0):
        bank.depth[j] = torch.from_numpy(wl.depth_of(j)).cuda()
    k = len(slots)
    S = k * wl.F
    n = wl.Nq * S
    idx = torch.tensor(np.asarray(slots, dtype=np.int32), device="cuda")
    cnt = torch.tensor([count], dtype=torch.int32, device="cuda")
    dcur = torch.from_numpy(wl.depth_of(wl.n)).cuda()
    uv_buf = torch.full((2 * n + 2,), -9.0, device="cuda")
    cell_buf = torch.full((n + 1,), -9, dtype=torch.int32, device="cuda")
    valid_buf = torch.full((n + 1,), 9, dtype=torch.uint8, device="cuda")
    uv, cell, valid = uv_buf[2:].view(wl.Nq, S, 2), cell_buf[1:].view(wl.Nq, S), valid_buf[1:].view(wl.Nq, S)
    assert uv.data_ptr() % 16 == 8 and cell.data_ptr() % 8 == 4 and valid.data_ptr() % 2 == 1
    api.crc_correspond(shp, synth.frame_records(wl.cur_frames), dcur, bank, idx, cnt, k, 0.05, uv, cell, valid)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(uv.cpu().numpy().astype(np.float64), ref[0])
    np.testing.assert_array_equal(cell.cpu().numpy(), ref[1])
    np.testing.assert_array_equal(valid.cpu().numpy(), ref[2])
    assert uv_buf[:2].eq(-9.0).all() and cell_buf[0].item() == -9 and valid_buf[0].item() == 9  # nothing outside
    uv2 = torch.full((wl.Nq, S, 2), -9.0, device="cuda")
    valid2 = torch.full((wl.Nq, S), 9, dtype=torch.uint8, device="cuda")
    api.crc_correspond(shp, synth.frame_records(wl.cur_frames), dcur, bank, idx, cnt, k, 0.05, uv2, None, valid2)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(uv2.cpu().numpy().astype(np.float64), ref[0])
    np.testing.assert_array_equal(valid2.cpu().numpy(), ref[2])
