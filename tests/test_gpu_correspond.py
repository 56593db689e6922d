"""GPU parity of the reprojection correspondence (Eq. 3-4) against the oracle.

Landing cells and valid flags must be identical except for pairs whose integer
decision lies within rounding distance of a boundary (u^ + 1/2 within 1e-4 of an
integer, or the depth / visibility comparison within 1e-6 / 1e-5 relative);
u^ of pairs valid on both sides must agree to 1e-3 token."""

import math

import numpy as np
import pytest
import torch

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
