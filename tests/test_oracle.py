"""Pins for the fp64 oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: hand-worked
retrieval scores (Eq. 1), the identity warp, the pure-translation closed form
and the pure-rotation homography of Eq. 3, an analytic ray-cast scene, a
brute-force double-loop softmax, torch's SDPA as a library routine, and the
statements the paper makes about the bias of Eq. 2 (non-positive, zero at the
correspondence, a multiplicative factor exp(lambda B) on the weights, exact
fallback for invalid queries).
"""

import json
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _f(x):
    return math.inf if x == "inf" else float(x)


# ----------------------------------------------------------------------------
# chunk pose (Sec. 4.2)
# ----------------------------------------------------------------------------


def test_chunk_pose_mean_centre_and_axis():
    R = np.stack([synth.camera_rotation(0.0), synth.camera_rotation(0.0), synth.camera_rotation(0.0)])
    c = np.array([[0.0, 0.0, 0.0], [3.0, 0.0, 0.0], [0.0, 3.0, 0.0]])
    centre, view = oracle.chunk_pose(R, c)
    np.testing.assert_allclose(centre, [1.0, 1.0, 0.0], atol=1e-15)
    np.testing.assert_allclose(view, [1.0, 0.0, 0.0], atol=1e-15)
    # two frames looking along +x and +y: the chunk looks along the bisector
    R2 = np.stack([synth.camera_rotation(0.0), synth.camera_rotation(math.pi / 2)])
    _, v2 = oracle.chunk_pose(R2, np.zeros((2, 3)))
    np.testing.assert_allclose(v2, [math.sqrt(0.5), math.sqrt(0.5), 0.0], atol=1e-15)
    assert abs(np.linalg.norm(v2) - 1.0) < 1e-15


def test_chunk_pose_optical_axis_is_forward():
    # the camera looks along its +z axis, so a pitched camera's view direction climbs
    R = synth.camera_rotation(0.3, 0.2)[None]
    _, v = oracle.chunk_pose(R, np.zeros((1, 3)))
    np.testing.assert_allclose(v, [math.cos(0.2) * math.cos(0.3), math.cos(0.2) * math.sin(0.3), math.sin(0.2)],
                               atol=1e-15)


# ----------------------------------------------------------------------------
# retrieval (Eq. 1)
# ----------------------------------------------------------------------------


def _handworked():
    g = json.load(open(os.path.join(GOLDEN, "retrieval_handworked.json")))
    bank_c, bank_v = [], []
    for e in g["bank"]:
        c, v = oracle.chunk_pose(synth.camera_rotation(math.radians(e["yaw_deg"]))[None], np.array([e["c"]]))
        bank_c.append(c)
        bank_v.append(v)
    cn, vn = oracle.chunk_pose(synth.camera_rotation(math.radians(g["current"]["yaw_deg"]))[None],
                               np.array([g["current"]["c"]]))
    return g, np.array(bank_c), np.array(bank_v), cn, vn


def test_retrieval_handworked_golden():
    g, bc, bv, cn, vn = _handworked()
    for case in g["cases"]:
        idx, score, count = oracle.retrieve(bc, bv, cn, vn, g["n"], case["E"], g["w_v"], _f(case["tau_c"]),
                                            case["cos_tau_v"], case["delta"], case["k"])
        assert count == case["count"], case
        assert list(idx) == case["idx"], case
        exp = np.array([_f(s) for s in case["score"]])
        fin = np.isfinite(exp)
        np.testing.assert_allclose(score[fin], exp[fin], rtol=0, atol=1e-12)
        assert np.all(np.isinf(score[~fin]))


def test_retrieval_gates_flip_at_threshold():
    # one candidate at distance exactly 2 and angle exactly 90 deg, gap exactly 5
    bc = np.array([[2.0, 0.0, 0.0]])
    bv = np.array([[0.0, 1.0, 0.0]])
    cn = np.zeros(3)
    vn = np.array([1.0, 0.0, 0.0])
    args = dict(E=1.0, w_v=0.5, k=1)
    assert oracle.retrieve(bc, bv, cn, vn, 5, tau_c=2.0, cos_tau_v=0.0, delta=5, **args)[2] == 1
    assert oracle.retrieve(bc, bv, cn, vn, 5, tau_c=np.nextafter(2.0, 0), cos_tau_v=0.0, delta=5, **args)[2] == 0
    assert oracle.retrieve(bc, bv, cn, vn, 5, tau_c=2.0, cos_tau_v=1e-300, delta=5, **args)[2] == 0
    assert oracle.retrieve(bc, bv, cn, vn, 5, tau_c=2.0, cos_tau_v=0.0, delta=6, **args)[2] == 0
    # E scales only the distance term: s = 2/E + 0.5 * (1 - 0)
    _, s, _ = oracle.retrieve(bc, bv, cn, vn, 5, E=4.0, w_v=0.5, tau_c=math.inf, cos_tau_v=-1.0, delta=0, k=1)
    assert s[0] == 0.5 + 0.5


def test_exclude_sink_removes_only_the_anchor_chunk():
    # chunk 0 is the best match; chunk 2 the second best (Sec. 4.2: the anchor is always in the cache)
    bc = np.array([[0.1, 0.0, 0.0], [5.0, 0.0, 0.0], [0.2, 0.0, 0.0]])
    bv = np.tile([1.0, 0.0, 0.0], (3, 1))
    args = (np.zeros(3), np.array([1.0, 0.0, 0.0]), 10, 1.0, 0.5, math.inf, -1.0, 1, 2)
    idx, _, count = oracle.retrieve(bc, bv, *args)
    assert count == 2 and list(idx) == [0, 2]
    idx, _, count = oracle.retrieve(bc, bv, *args, exclude_sink=True)
    assert count == 2 and list(idx) == [2, 1]


def test_retrieval_ties_break_by_chunk_index():
    bc = np.array([[1.0, 0, 0], [0, 1.0, 0], [1.0, 0, 0], [0, 0, 1.0]])
    bv = np.tile([1.0, 0.0, 0.0], (4, 1))
    idx, _, count = oracle.retrieve(bc, bv, np.zeros(3), np.array([1.0, 0, 0]), 10, 1.0, 0.5, math.inf, -1.0, 1, 4)
    assert count == 4 and list(idx) == [0, 1, 2, 3]


def test_retrieval_permutation_invariance():
    g = np.random.default_rng(7)
    bc = g.normal(size=(50, 3)) * 5
    bv = g.normal(size=(50, 3))
    bv /= np.linalg.norm(bv, axis=1, keepdims=True)
    cn = g.normal(size=3)
    vn = np.array([0.0, 0.0, 1.0])
    idx, score, _ = oracle.retrieve(bc, bv, cn, vn, 100, 3.0, 0.5, math.inf, -1.0, 1, 5)
    perm = g.permutation(50)
    idx2, score2, _ = oracle.retrieve(bc[perm], bv[perm], cn, vn, 100, 3.0, 0.5, math.inf, -1.0, 1, 5)
    assert list(perm[idx2]) == list(idx)
    np.testing.assert_array_equal(score, score2)


def test_empty_admissible_set_extends_window():
    # Sec. 4.2: with A_n empty the retrieved slot extends the recent window
    idx = np.array([-1, -1], dtype=np.int32)
    assert list(oracle.fill_slots(idx, 0, ext_first=7, ext_min=1)) == [7, 6]
    assert list(oracle.fill_slots(np.array([4, -1], dtype=np.int32), 1, ext_first=7, ext_min=1)) == [4, 7]
    assert list(oracle.fill_slots(idx, 0, ext_first=1, ext_min=1)) == [1, -1]
    assert list(oracle.fill_slots(idx, 0, ext_first=-1, ext_min=1)) == [-1, -1]


def test_retrieval_over_resident_chunks_equals_retrieval_over_that_sub_bank():
    # a chunk whose keys and values are no longer held is not admissible: the result is that of
    # Eq. 1 over the bank with those chunks removed (brute force on the sub-bank, indices mapped back)
    g = np.random.default_rng(8)
    bc = g.normal(size=(40, 3)) * 4
    bv = g.normal(size=(40, 3))
    bv /= np.linalg.norm(bv, axis=1, keepdims=True)
    cn, vn = g.normal(size=3), np.array([0.0, 1.0, 0.0])
    resident = g.uniform(size=40) < 0.5
    args = (cn, vn, 100, 2.0, 0.5, math.inf, -1.0, 1, 6)
    idx, score, count = oracle.retrieve(bc, bv, *args, resident=resident)
    keep = np.nonzero(resident)[0]
    idx2, score2, count2 = oracle.retrieve(bc[keep], bv[keep], *args)
    assert count == count2 == 6
    assert list(idx) == list(keep[idx2])
    np.testing.assert_array_equal(score, score2)
    assert resident[idx[:count]].all()
    # every chunk resident: the literal Eq. 1
    full = oracle.retrieve(bc, bv, *args)
    assert list(oracle.retrieve(bc, bv, *args, resident=np.ones(40, bool))[0]) == list(full[0])
    # the window-extension fallback skips a chunk that is no longer held
    res = np.ones(10, bool)
    res[6] = False
    assert list(oracle.fill_slots(np.array([-1, -1], dtype=np.int32), 0, 7, 1, resident=res)) == [7, -1]
    assert list(oracle.fill_slots(np.array([-1, -1], dtype=np.int32), 0, 6, 1, resident=res)) == [-1, 5]


def test_gather_is_slab_copy():
    pool = np.arange(4 * 2 * 1 * 3 * 1 * 2, dtype=np.float32).reshape(4, 2, 1, 3, 1, 2)
    out = oracle.gather(pool, np.array([5, -1, 2]), 4)
    np.testing.assert_array_equal(out[0], pool[1])
    assert out[1] is None
    np.testing.assert_array_equal(out[2], pool[2])


# ----------------------------------------------------------------------------
# correspondence (Eq. 3-4)
# ----------------------------------------------------------------------------


def _grid_u(h, w):
    ii, jj = np.meshgrid(np.arange(h, dtype=np.float64), np.arange(w, dtype=np.float64), indexing="ij")
    return np.stack([jj.ravel(), ii.ravel()], axis=1)


def _one(R, c, K):
    return K[None], R[None], np.asarray(c, dtype=np.float64)[None]


def test_identity_pose_maps_token_to_itself():
    h, w = 6, 9
    K = synth.pinhole(h, w, 70.0)
    R = synth.random_rotation(np.random.default_rng(1), 180.0)
    c = np.array([0.3, -2.0, 1.0])
    dep = np.exp(np.random.default_rng(2).uniform(-1, 3, size=(1, h, w)))
    Kt, Rt, ct = _one(R, c, K)
    uv, cell, valid = oracle.correspond(dep, Kt, Rt, ct, dep, Kt, Rt, ct, eps=0.05)
    np.testing.assert_allclose(uv[:, 0], _grid_u(h, w), atol=1e-12)
    assert valid.all()
    np.testing.assert_array_equal(cell[:, 0], np.arange(h * w))


def test_pure_translation_closed_form():
    # R_s = R_t = R; Delta = R^T (c_t - c_s) in camera axes:
    # x^ = c_x + (z (j - c_x) + f Delta_x) / (z + Delta_z), likewise for y.
    g = np.random.default_rng(3)
    h, w = 7, 11
    K = synth.pinhole(h, w, 90.0)
    f, cx, cy = K[0, 0], K[0, 2], K[1, 2]
    R = synth.random_rotation(g, 180.0)
    ct = g.normal(size=3)
    cs = ct + g.normal(size=3) * 0.3
    dep = np.exp(g.uniform(0, 3, size=(1, h, w)))
    Kt, Rt, ctt = _one(R, ct, K)
    _, Rs, css = _one(R, cs, K)
    uv, _, _ = oracle.correspond(dep, Kt, Rt, ctt, dep, Kt, Rs, css, eps=math.inf)
    D = R.T @ (ct - cs)
    u = _grid_u(h, w)
    z = dep[0].ravel()
    xs = cx + (z * (u[:, 0] - cx) + f * D[0]) / (z + D[2])
    ys = cy + (z * (u[:, 1] - cy) + f * D[1]) / (z + D[2])
    np.testing.assert_allclose(uv[:, 0, 0], xs, rtol=0, atol=1e-9)
    np.testing.assert_allclose(uv[:, 0, 1], ys, rtol=0, atol=1e-9)


def test_lateral_translation_is_disparity():
    h, w = 5, 8
    K = synth.pinhole(h, w, 90.0)
    R = synth.camera_rotation(0.4)
    dep = np.full((1, h, w), 4.0)
    right = R[:, 0]
    Kt, Rt, ct = _one(R, np.zeros(3), K)
    # source camera 0.5 m to the left of the target: points shift right by f * 0.5 / z
    uv, _, _ = oracle.correspond(dep, Kt, Rt, ct, dep, Kt, Rt, (-0.5 * right)[None], eps=math.inf)
    np.testing.assert_allclose(uv[:, 0, 0] - _grid_u(h, w)[:, 0], K[0, 0] * 0.5 / 4.0, atol=1e-12)
    np.testing.assert_allclose(uv[:, 0, 1], _grid_u(h, w)[:, 1], atol=1e-12)


def test_pure_rotation_is_depth_free_homography():
    # Sec. 4.3: with c_s = c_t depth cancels and Eq. 3 is pi(K_s R_s^T R_t K_t^-1 u~)
    g = np.random.default_rng(4)
    h, w = 9, 13
    Kt = synth.pinhole(h, w, 90.0)
    Ks = synth.pinhole(h, w, 60.0)  # zoom
    Rt = synth.random_rotation(g, 180.0)
    Rs = Rt @ synth.random_rotation(g, 20.0)
    c = g.normal(size=3)
    d1 = np.exp(g.uniform(-1, 4, size=(1, h, w)))
    d2 = np.exp(g.uniform(-1, 4, size=(1, h, w)))
    a = oracle.correspond(d1, Kt[None], Rt[None], c[None], d1, Ks[None], Rs[None], c[None], math.inf)[0]
    b = oracle.correspond(d2, Kt[None], Rt[None], c[None], d2, Ks[None], Rs[None], c[None], math.inf)[0]
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-9)
    Hm = Ks @ Rs.T @ Rt @ np.linalg.inv(Kt)
    u = _grid_u(h, w)
    q = (Hm @ np.concatenate([u, np.ones((h * w, 1))], axis=1).T).T
    np.testing.assert_allclose(a[:, 0], q[:, :2] / q[:, 2:], rtol=0, atol=1e-9)


def test_reprojection_matches_analytic_scene_and_round_trips():
    g = synth.rng(5, "scene")
    scene = synth.Scene.room(g, radius=20.0, n_walls=8, n_boards=12, board_rmin=3.0, board_rmax=15.0)
    h, w = 12, 20
    K = synth.pinhole(h, w, 90.0)
    Rt = synth.camera_rotation(0.2, 0.05)
    ct = np.array([1.0, 0.5, 1.6])
    Rs = synth.camera_rotation(0.5, -0.05)
    cs = np.array([0.2, 1.8, 1.5])
    zt = synth.render_depth(scene, K, Rt, ct, h, w, 1e-6, 1e6)
    u = _grid_u(h, w)
    uh, Xs = oracle.reproject(u, zt.ravel(), K, Rt, ct, K, Rs, cs)
    front = Xs[:, 2] > 1e-6
    assert front.sum() > 100
    # the scene point lies on the source ray through u^ at depth [X_s]_z: the first hit
    # along that ray is never farther, and equals it wherever the point is visible
    hit = synth.render_depth(scene, K, Rs, cs, h, w, 1e-6, 1e6, pix=uh[front])
    assert np.all(hit <= Xs[front, 2] * (1 + 1e-9) + 1e-9)
    vis = np.abs(hit - Xs[front, 2]) <= 1e-7 * Xs[front, 2]
    assert vis.mean() > 0.5
    # warping back from s to t with the point's own source depth returns u_p and z_p
    ub, Xt = oracle.reproject(uh[front], Xs[front, 2], K, Rs, cs, K, Rt, ct)
    np.testing.assert_allclose(ub, u[front], atol=1e-9)
    np.testing.assert_allclose(Xt[:, 2], zt.ravel()[front], rtol=1e-12)


def test_visibility_rejects_occluded_points():
    # target sees a wall at z = 10; the source camera is 1 m to the right and a
    # source-side occluder at depth 2 covers columns 0..3: points landing there fail Eq. 4
    h, w = 6, 10
    K = synth.pinhole(h, w, 90.0)
    R = np.eye(3)
    dt = np.full((1, h, w), 10.0)
    ds = np.full((1, h, w), 10.0)
    ds[0, :, :4] = 2.0
    uv, cell, valid = oracle.correspond(dt, K[None], R[None], np.zeros((1, 3)), ds, K[None], R[None],
                                        np.array([[1.0, 0.0, 0.0]]), eps=0.05)
    x = np.floor(uv[:, 0, 0] + 0.5)
    inb = (x >= 0) & (x < w)
    np.testing.assert_array_equal(valid[:, 0], inb & (x >= 4))
    # eps = +inf disables the test
    _, _, v2 = oracle.correspond(dt, K[None], R[None], np.zeros((1, 3)), ds, K[None], R[None],
                                 np.array([[1.0, 0.0, 0.0]]), eps=math.inf)
    np.testing.assert_array_equal(v2[:, 0], inb)
    # eps is a relative tolerance: depth 10 vs source 9.6 passes with 5 %, fails with 1 %
    ds2 = np.full((1, h, w), 9.6)
    a = oracle.correspond(dt, K[None], R[None], np.zeros((1, 3)), ds2, K[None], R[None], np.zeros((1, 3)), 0.05)[2]
    b = oracle.correspond(dt, K[None], R[None], np.zeros((1, 3)), ds2, K[None], R[None], np.zeros((1, 3)), 0.01)[2]
    assert a.all() and not b.any()


def test_behind_camera_off_grid_and_bad_depth_are_invalid():
    h, w = 4, 6
    K = synth.pinhole(h, w, 90.0)
    dep = np.full((1, h, w), 3.0)
    Rt = synth.camera_rotation(0.0)
    Rs = synth.camera_rotation(math.pi)  # looks backwards
    c = np.zeros((1, 3))
    assert not oracle.correspond(dep, K[None], Rt[None], c, dep, K[None], Rs[None], c, math.inf)[2].any()
    far = (100.0 * Rt[:, 0])[None]  # 100 m to the side: lands off the grid
    assert not oracle.correspond(dep, K[None], Rt[None], c, dep, K[None], Rt[None], far, math.inf)[2].any()
    bad = dep.copy()
    bad[0, 0, :3] = [0.0, -1.0, np.nan]
    v = oracle.correspond(bad, K[None], Rt[None], c, dep, K[None], Rt[None], c, math.inf)[2][:, 0]
    assert not v[:3].any() and v[3:].all()
    # a frame whose slot holds no retrieved chunk carries no correspondence
    v = oracle.correspond(dep, K[None], Rt[None], c, dep, K[None], Rt[None], c, math.inf,
                          source_ok=np.array([False]))[2]
    assert not v.any()


def test_landing_cell_rounds_half_up():
    # u^ lands exactly half way between columns 1 and 2: cell = floor(x + 1/2) = 2
    h, w = 3, 4
    K = np.array([[2.0, 0.0, 1.5], [0.0, 2.0, 1.0], [0.0, 0.0, 1.0]])  # f = 2, exact in binary
    dep = np.full((1, h, w), 4.0)
    R = np.eye(3)
    # shift by f * t / z = 0.5 column: t = 1
    uv, cell, valid = oracle.correspond(dep, K[None], R[None], np.zeros((1, 3)), dep, K[None], R[None],
                                        np.array([[-1.0, 0.0, 0.0]]), math.inf)
    assert uv[1, 0, 0] == 1.5 and cell[1, 0] == 2
    assert not valid[3, 0] and valid[2, 0]  # column 3 + 0.5 rounds to 4 = off grid


# ----------------------------------------------------------------------------
# attention (Eq. 2)
# ----------------------------------------------------------------------------


def _tiny_attn_inputs(seed=0, h=2, w=3, F=2, d=8, with_ret=True):
    g = np.random.default_rng(seed)
    Nc = F * h * w
    segs = [(0, Nc, oracle.crc_oracle.SEG_SINK, 0), (Nc, Nc, oracle.crc_oracle.SEG_RETRIEVED, 0),
            (2 * Nc, Nc, oracle.crc_oracle.SEG_WINDOW, 0)]
    Nk = 3 * Nc
    Q = g.normal(size=(1, Nc, 1, d))
    Kc = g.normal(size=(1, Nk, 1, d))
    Vc = g.normal(size=(1, Nk, 1, d))
    uv = g.uniform(-0.5, max(h, w), size=(Nc, F, 2))
    valid = g.uniform(size=(Nc, F)) < 0.7
    return Q, Kc, Vc, uv, valid, segs, h, w, F


def _brute(Q, Kc, Vc, bias_fn):
    """Naive double loop softmax attention (one layer, one head)."""
    Nq, d = Q.shape[1], Q.shape[3]
    out = np.zeros((Nq, d))
    lse = np.zeros(Nq)
    for p in range(Nq):
        logits = []
        for kk in range(Kc.shape[1]):
            dot = 0.0
            for e in range(d):
                dot += Q[0, p, 0, e] * Kc[0, kk, 0, e]
            logits.append(dot / math.sqrt(d) + bias_fn(p, kk))
        m = max(logits)
        ex = [math.exp(a - m) for a in logits]
        ssum = sum(ex)
        for e in range(d):
            out[p, e] = sum(ex[kk] * Vc[0, kk, 0, e] for kk in range(len(ex))) / ssum
        lse[p] = m + math.log(ssum)
    return out, lse


def test_lambda_zero_is_plain_softmax_attention_bruteforce():
    Q, Kc, Vc, uv, valid, segs, h, w, F = _tiny_attn_inputs()
    O, lse = oracle.attention(Q, Kc, Vc, uv, valid, segs, h, w, F, lam=0.0, sigma=1.0)
    Ob, lb = _brute(Q, Kc, Vc, lambda p, k: 0.0)
    np.testing.assert_allclose(O[0, :, 0], Ob, atol=1e-12)
    np.testing.assert_allclose(lse[0, 0], lb, atol=1e-12)


def test_lambda_zero_matches_library_sdpa():
    torch = pytest.importorskip("torch")
    g = np.random.default_rng(11)
    L, Nq, H, d, Nk = 2, 24, 3, 16, 40
    Q, Kc, Vc = g.normal(size=(L, Nq, H, d)), g.normal(size=(L, Nk, H, d)), g.normal(size=(L, Nk, H, d))
    segs = [(0, Nk, oracle.crc_oracle.SEG_WINDOW, 0)]
    O, _ = oracle.attention(Q, Kc, Vc, np.zeros((Nq, 1, 2)), np.zeros((Nq, 1), bool), segs, 1, 1, 1, 0.0, 1.0)
    t = lambda a: torch.from_numpy(a).permute(0, 2, 1, 3)  # noqa: E731  [L, H, N, d]
    ref = torch.nn.functional.scaled_dot_product_attention(t(Q), t(Kc), t(Vc)).permute(0, 2, 1, 3).numpy()
    np.testing.assert_allclose(O, ref, atol=1e-12)


def test_all_invalid_queries_reduce_exactly_to_plain_attention():
    Q, Kc, Vc, uv, valid, segs, h, w, F = _tiny_attn_inputs(seed=2)
    O0, l0 = oracle.attention(Q, Kc, Vc, uv, valid, segs, h, w, F, lam=0.0, sigma=1.0)
    O1, l1 = oracle.attention(Q, Kc, Vc, uv, np.zeros_like(valid), segs, h, w, F, lam=5.0, sigma=0.7)
    np.testing.assert_array_equal(O0, O1)
    np.testing.assert_array_equal(l0, l1)


def test_bias_is_multiplicative_suppression_factor():
    # Sec. 4.3: the bias multiplies each retrieved key's weight by exp(lambda B) in (0, 1];
    # weights with bias = weights without bias x exp(lambda B), renormalised.
    torch = pytest.importorskip("torch")
    Q, Kc, Vc, uv, valid, segs, h, w, F = _tiny_attn_inputs(seed=3)
    lam, sigma = 1.7, 0.8
    Nc = F * h * w
    # identity values expose the softmax weights: O = weights
    Nk = Kc.shape[1]
    Vid = np.eye(Nk)[None, :, None, :]
    Kp = np.concatenate([Kc, np.zeros((1, Nk, 1, Nk - Kc.shape[3]))], axis=3)
    Qp = np.concatenate([Q, np.zeros((1, Nc, 1, Nk - Q.shape[3]))], axis=3)
    W0, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=0.0, sigma=sigma)
    W1, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=lam, sigma=sigma)
    W0, W1 = W0[0, :, 0], W1[0, :, 0]
    # the Gaussian factor at each retrieved key, from grid geometry
    fac = np.ones((Nc, Nk))
    for loc in range(Nc):
        s, rem = divmod(loc, h * w)
        y, x = divmod(rem, w)
        dist2 = (x - uv[:, s, 0]) ** 2 + (y - uv[:, s, 1]) ** 2
        fac[:, Nc + loc] = np.where(valid[:, s], np.exp(-lam * dist2 / (2 * sigma * sigma)), 1.0)
    assert np.all(fac <= 1.0) and np.all(fac > 0.0)
    expect = W0 * fac
    expect /= expect.sum(axis=1, keepdims=True)
    np.testing.assert_allclose(W1, expect, atol=1e-13)
    # and the library SDPA with the additive mask log(fac) agrees
    t = lambda a: torch.from_numpy(a).permute(0, 2, 1, 3)  # noqa: E731
    ref = torch.nn.functional.scaled_dot_product_attention(
        t(Qp), t(Kp), t(Vid), attn_mask=torch.from_numpy(np.log(fac))[None, None], scale=1.0 / math.sqrt(Qp.shape[3]))
    np.testing.assert_allclose(W1, ref.permute(0, 2, 1, 3).numpy()[0, :, 0], atol=1e-13)


def test_bias_vanishes_at_correspondence_and_concentrates_as_lambda_grows():
    h, w, F, d = 3, 4, 2, 4
    Nc = F * h * w
    segs = [(0, Nc, 0, 0), (Nc, Nc, 1, 0)]
    Nk = 2 * Nc
    Q = np.zeros((1, Nc, 1, d))
    Kc = np.zeros((1, Nk, 1, d))  # all logits equal without bias
    Vid = np.eye(Nk)[None, :, None, :]
    Kp = np.zeros((1, Nk, 1, Nk))
    Qp = np.zeros((1, Nc, 1, Nk))
    uv = np.zeros((Nc, F, 2))
    valid = np.zeros((Nc, F), bool)
    # query 0 corresponds to source frame 1, cell (x=2, y=1) exactly
    uv[0, 1] = (2.0, 1.0)
    valid[0, 1] = True
    target = Nc + 1 * h * w + 1 * w + 2
    Wl, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=1.0, sigma=1.0)
    W0, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=0.0, sigma=1.0)
    # zero bias at u^: the weight ratio of the matching key to a sink key is unchanged
    assert Wl[0, 0, 0, target] / Wl[0, 0, 0, 0] == pytest.approx(W0[0, 0, 0, target] / W0[0, 0, 0, 0], rel=1e-14)
    # a neighbour one cell away in x is suppressed by exactly exp(-lambda / (2 sigma^2))
    assert Wl[0, 0, 0, target - 1] / Wl[0, 0, 0, target] == pytest.approx(math.exp(-0.5), rel=1e-14)
    # keys of the other source frame (frame 0) are biased too: query 0 has no valid pair there
    assert Wl[0, 0, 0, Nc] == pytest.approx(Wl[0, 0, 0, 0], rel=1e-14)
    # as lambda grows the retrieved mass concentrates on the nearest key
    Wb, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=200.0, sigma=1.0)
    ret = Wb[0, 0, 0, Nc + h * w:2 * Nc]
    assert ret.argmax() == 1 * w + 2 and ret.max() / ret.sum() > 1 - 1e-12
    # other queries (no valid correspondence) are untouched
    np.testing.assert_array_equal(Wb[0, 1:], W0[0, 1:])


def test_additive_gaussian_form_raises_weights_near_the_correspondence():
    # opt-in variant: A = q.k/sqrt(d) + beta exp(-d^2 / (2 sigma^2)) on retrieved keys with a valid pair
    h, w, F = 3, 4, 2
    Nc = F * h * w
    segs = [(0, Nc, 0, 0), (Nc, Nc, 1, 0)]
    Nk = 2 * Nc
    Vid = np.eye(Nk)[None, :, None, :]
    Kp = np.zeros((1, Nk, 1, Nk))
    Qp = np.zeros((1, Nc, 1, Nk))  # all logits equal without bias
    uv = np.zeros((Nc, F, 2))
    valid = np.zeros((Nc, F), bool)
    uv[0, 1] = (2.0, 1.0)
    valid[0, 1] = True
    target = Nc + 1 * h * w + 1 * w + 2
    beta, sigma = 1.3, 0.9
    Wg, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=beta, sigma=sigma, bias_form="gaussian")
    # at the correspondence the weight is e^beta times a sink key's
    assert Wg[0, 0, 0, target] / Wg[0, 0, 0, 0] == pytest.approx(math.exp(beta), rel=1e-14)
    # one cell away: e^(beta exp(-1 / (2 sigma^2)))
    assert Wg[0, 0, 0, target - 1] / Wg[0, 0, 0, 0] == pytest.approx(
        math.exp(beta * math.exp(-1.0 / (2 * sigma * sigma))), rel=1e-14)
    # the other source frame (no valid pair for query 0) and the other queries are untouched
    assert Wg[0, 0, 0, Nc] == pytest.approx(Wg[0, 0, 0, 0], rel=1e-14)
    W0, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=0.0, sigma=sigma, bias_form="gaussian")
    np.testing.assert_array_equal(Wg[0, 1:], W0[0, 1:])
    # far from the correspondence the bonus vanishes: a 1 x 40 frame, keys 30 cells away
    h2, w2, F2 = 1, 40, 1
    segs2 = [(0, 40, 0, 0), (40, 40, 1, 0)]
    uv2 = np.zeros((40, 1, 2))
    valid2 = np.ones((40, 1), bool)
    W2, _ = oracle.attention(np.zeros((1, 40, 1, 80)), np.zeros((1, 80, 1, 80)), np.eye(80)[None, :, None, :],
                             uv2, valid2, segs2, h2, w2, F2, lam=beta, sigma=1.0, bias_form="gaussian")
    assert W2[0, 0, 0, 40 + 30] / W2[0, 0, 0, 0] == pytest.approx(1.0, abs=1e-12)
    with pytest.raises(ValueError):
        oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=beta, sigma=sigma, bias_form="other")


def test_empty_retrieved_slot_is_masked():
    Q, Kc, Vc, uv, valid, segs, h, w, F = _tiny_attn_inputs(seed=5)
    Nc = F * h * w
    O, _ = oracle.attention(Q, Kc, Vc, uv, valid, segs, h, w, F, lam=2.0, sigma=1.0,
                            slot_chunks=np.array([-1]))
    keep = np.r_[0:Nc, 2 * Nc:3 * Nc]
    Ob, _ = _brute(Q, Kc[:, keep], Vc[:, keep], lambda p, k: 0.0)
    np.testing.assert_allclose(O[0, :, 0], Ob, atol=1e-12)
    # a zero-length window segment is simply absent
    segs2 = segs[:2] + [(2 * Nc, 0, 2, 0)]
    O2, _ = oracle.attention(Q, Kc, Vc, uv, np.zeros_like(valid), segs2, h, w, F, lam=2.0, sigma=1.0)
    Ob2, _ = _brute(Q, Kc[:, :2 * Nc], Vc[:, :2 * Nc], lambda p, k: 0.0)
    np.testing.assert_allclose(O2[0, :, 0], Ob2, atol=1e-12)


def test_paper_constants_match_workload_shapes():
    c = json.load(open(os.path.join(GOLDEN, "paper_constants.json")))
    wl = synth.make_workload(2)
    assert (wl.F, wl.h, wl.w) == (c["F"], c["h"], c["w"])
    frames = [length // (wl.h * wl.w) for _, length, _, _ in wl.segments]
    assert sum(frames) == c["M_frames"]
    assert frames[0] == c["anchor_frames"] and frames[1] == c["retrieved_frames"]
    assert sum(frames[2:]) == c["recent_frames"]
    assert wl.w_v == c["w_v"]


def test_source_frame_index_spans_slots():
    # with two retrieved slots of F frames each, source frame s = slot * F + frame:
    # a correspondence in s = 3 (slot 1, frame 1) must pull weight onto that block only
    h, w, F = 2, 3, 2
    Nc = F * h * w
    segs = [(0, Nc, 0, 0), (Nc, Nc, 1, 0), (2 * Nc, Nc, 1, 1)]
    Nk = 3 * Nc
    Vid = np.eye(Nk)[None, :, None, :]
    Qp = np.zeros((1, Nc, 1, Nk))
    Kp = np.zeros((1, Nk, 1, Nk))
    uv = np.zeros((Nc, 2 * F, 2))
    valid = np.zeros((Nc, 2 * F), bool)
    uv[0, 3] = (1.0, 1.0)
    valid[0, 3] = True
    W, _ = oracle.attention(Qp, Kp, Vid, uv, valid, segs, h, w, F, lam=100.0, sigma=1.0)
    blk = W[0, 0, 0, 2 * Nc + h * w:]
    assert blk.argmax() == 1 * w + 1 and blk.max() == pytest.approx(W[0, 0, 0, 0], rel=1e-14)
    # slot 0 and the first frame of slot 1 are not biased for query 0
    np.testing.assert_allclose(W[0, 0, 0, Nc:2 * Nc + h * w], W[0, 0, 0, 0], rtol=1e-14)


# ----------------------------------------------------------------------------
# RoPE re-positioning of a re-packed chunk (Sec. 4.2 "Cache packing")
# ----------------------------------------------------------------------------


def _rotary(x, pos, channel0, pairs, theta, interleaved):
    """Standard rotary embedding written with explicit 2x2 rotation matrices: pair i of
    a token at position pos is rotated by the angle pos * theta^(-i/pairs)."""
    out = np.array(x, dtype=np.float64)
    pos = np.asarray(pos, dtype=np.float64)
    for i in range(pairs):
        a, b = (channel0 + 2 * i, channel0 + 2 * i + 1) if interleaved else (channel0 + i, channel0 + i + pairs)
        ang = pos * theta ** (-i / pairs)
        ca, sa = np.cos(ang), np.sin(ang)
        xa, xb = out[..., a].copy(), out[..., b].copy()
        out[..., a] = ca * xa - sa * xb
        out[..., b] = sa * xa + ca * xb
    return out


def test_rope_handworked_quarter_turn_and_frequency():
    # pair 0 has frequency 1: a shift of 1 rotates (1, 0) by one radian, counter-clockwise
    x = np.array([1.0, 0.0, 0.3, 0.7])
    y = oracle.rope_reposition(x, 1, 0, 2, 4.0 / math.pi ** 2, True)
    assert abs(y[0] - 0.5403023058681398) < 1e-15 and abs(y[1] - 0.8414709848078965) < 1e-15
    # pair 1 has frequency theta^(-1/2) = pi/2 for theta = 4/pi^2: a quarter turn (a, b) -> (-b, a)
    assert abs(y[2] + 0.7) < 1e-15 and abs(y[3] - 0.3) < 1e-15
    # half-split layout: pair 0 = channels (0, 2), pair 1 = channels (1, 3)
    z = oracle.rope_reposition(np.array([1.0, 0.3, 0.0, 0.7]), 1, 0, 2, 4.0 / math.pi ** 2, False)
    assert abs(z[0] - 0.5403023058681398) < 1e-15 and abs(z[2] - 0.8414709848078965) < 1e-15
    assert abs(z[1] + 0.7) < 1e-15 and abs(z[3] - 0.3) < 1e-15


@pytest.mark.parametrize("interleaved", [True, False])
def test_rope_reposition_equals_embedding_at_new_position(interleaved):
    g = np.random.default_rng(3)
    d, c0, pairs, theta = 32, 8, 8, 10000.0
    k = g.normal(size=(5, d))
    q = g.normal(size=(5, d))
    for t, delta in ((7, 5), (40, -33), (3, 0)):
        moved = oracle.rope_reposition(_rotary(k, t, c0, pairs, theta, interleaved), delta, c0, pairs, theta,
                                       interleaved)
        np.testing.assert_allclose(moved, _rotary(k, t + delta, c0, pairs, theta, interleaved), atol=1e-12)
        # relative positions: moving the key by delta equals moving the query by -delta
        m = 11
        lhs = np.sum(_rotary(q, m, c0, pairs, theta, interleaved) * moved, axis=-1)
        rhs = np.sum(_rotary(q, m - delta, c0, pairs, theta, interleaved) * _rotary(k, t, c0, pairs, theta,
                                                                                   interleaved), axis=-1)
        np.testing.assert_allclose(lhs, rhs, atol=1e-12)
        # channels outside the temporal block are untouched; pair norms are kept
        outside = np.r_[0:c0, c0 + 2 * pairs:d]
        np.testing.assert_array_equal(moved[:, outside], k[:, outside])
        np.testing.assert_allclose(np.linalg.norm(moved, axis=-1), np.linalg.norm(k, axis=-1), rtol=1e-14)


def test_rope_reposition_composes_and_half_split_is_a_channel_permutation():
    g = np.random.default_rng(4)
    x = g.normal(size=(3, 16))
    a = oracle.rope_reposition(oracle.rope_reposition(x, 4, 0, 6, 500.0, True), -9, 0, 6, 500.0, True)
    np.testing.assert_allclose(a, oracle.rope_reposition(x, -5, 0, 6, 500.0, True), atol=1e-13)
    # half-split pair i = (c0 + i, c0 + i + pairs) is interleaved pair i after moving the channels
    c0, pairs = 2, 6
    perm = np.arange(16)
    perm[c0:c0 + 2 * pairs:2] = np.arange(c0, c0 + pairs)
    perm[c0 + 1:c0 + 2 * pairs:2] = np.arange(c0 + pairs, c0 + 2 * pairs)
    half = oracle.rope_reposition(x, 7, c0, pairs, 300.0, False)
    inter = oracle.rope_reposition(x[:, perm], 7, c0, pairs, 300.0, True)
    np.testing.assert_allclose(half[:, perm], inter, atol=1e-13)


def test_gather_repositions_keys_next_to_the_window():
    # keys cached with their rotary embedding at frame positions frame_pos0 + j F + f; after the
    # gather, slot r's frame f sits at pos_slot0 + r pos_stride + f.  Values are not rotated.
    g = np.random.default_rng(5)
    F, h, w, L, H, d, P = 2, 2, 3, 2, 2, 16, 4
    Nc = F * h * w
    frame = np.repeat(np.arange(F), h * w)[None, :, None]
    rope = dict(channel0=0, pairs=8, theta=10000.0, interleaved=True, pos_slot0=30, pos_stride=F, frame_pos0=-2,
                F=F)
    raw = g.normal(size=(P, 2, L, Nc, H, d))
    pool = raw.copy()
    chunks = [9, 6]  # chunk j lives in slab j % P
    for j in chunks:
        pool[j % P, 0] = _rotary(raw[j % P, 0], rope["frame_pos0"] + j * F + frame, 0, 8, 1e4, True)
    out = oracle.gather(pool, np.array(chunks + [-1]), P, rope=rope)
    for r, j in enumerate(chunks):
        want = _rotary(raw[j % P, 0], rope["pos_slot0"] + r * F + frame, 0, 8, 1e4, True)
        np.testing.assert_allclose(out[r][0], want, atol=1e-12)
        np.testing.assert_array_equal(out[r][1], pool[j % P, 1])
    assert out[2] is None


# ----------------------------------------------------------------------------
# frame-causal mask inside the current chunk (test mode of the attention)
# ----------------------------------------------------------------------------


def _frame_causal_case(seed=3, F=3, h=2, w=3):
    g = np.random.default_rng(seed)
    Nc = F * h * w
    segs = [(0, Nc, oracle.crc_oracle.SEG_SINK, 0), (Nc, Nc, oracle.crc_oracle.SEG_RETRIEVED, 0),
            (2 * Nc, Nc, oracle.crc_oracle.SEG_CURRENT, 0)]
    Nk = 3 * Nc
    Q = g.standard_normal((1, Nc, 1, 8))
    K = g.standard_normal((1, Nk, 1, 8))
    V = g.standard_normal((1, Nk, 1, 8))
    S = F
    uv = np.stack([g.uniform(0, w, (Nc, S)), g.uniform(0, h, (Nc, S))], -1)
    valid = g.uniform(size=(Nc, S)) < 0.7
    return Q, K, V, uv, valid, segs, (F, h, w)


def test_frame_causal_mask_matches_a_double_loop_softmax():
    Q, K, V, uv, valid, segs, (F, h, w) = _frame_causal_case()
    lam, sigma = 1.5, 0.8
    O, lse = oracle.attention(Q, K, V, uv, valid, segs, h, w, F, lam, sigma, mask_mode="frame")
    Nc, hw = F * h * w, h * w
    d = Q.shape[-1]
    for p in range(Nc):
        tq = p // hw
        logits, vals = [], []
        for kk in range(K.shape[1]):
            seg = kk // Nc
            loc = kk - seg * Nc
            if seg == 2 and loc // hw > tq:  # a later frame of the current chunk
                continue
            a = sum(Q[0, p, 0, e] * K[0, kk, 0, e] for e in range(d)) / math.sqrt(d)
            if seg == 1 and valid[p, loc // hw]:
                x, y = (loc % hw) % w, (loc % hw) // w
                ux, uy = uv[p, loc // hw]
                a += lam * -((x - ux) ** 2 + (y - uy) ** 2) / (2 * sigma * sigma)
            logits.append(a)
            vals.append(V[0, kk, 0])
        mx = max(logits)
        ex = [math.exp(a - mx) for a in logits]
        tot = sum(ex)
        ref = sum(e * v for e, v in zip(ex, vals)) / tot
        np.testing.assert_allclose(O[0, p, 0], ref, rtol=1e-12, atol=1e-12)
        assert lse[0, 0, p] == pytest.approx(mx + math.log(tot), abs=1e-12)


def test_frame_causal_mask_special_cases():
    # one frame per chunk: nothing to mask, the chunk mode exactly
    Q, K, V, uv, valid, segs, (F, h, w) = _frame_causal_case(seed=4, F=1, h=3, w=3)
    a = oracle.attention(Q, K, V, uv, valid, segs, h, w, F, 2.0, 1.0, mask_mode="frame")
    b = oracle.attention(Q, K, V, uv, valid, segs, h, w, F, 2.0, 1.0)
    np.testing.assert_array_equal(a[0], b[0])
    # only the current chunk: frame-0 queries attend to the frame-0 keys alone, the last frame's
    # queries to every key (the chunk mode)
    Q, K, V, uv, valid, _, (F, h, w) = _frame_causal_case(seed=5)
    Nc, hw = F * h * w, h * w
    cur = [(0, Nc, oracle.crc_oracle.SEG_CURRENT, 0)]
    O = oracle.attention(Q, K[:, :Nc], V[:, :Nc], uv, valid, cur, h, w, F, 2.0, 1.0, mask_mode="frame")[0]
    first = oracle.attention(Q[:, :hw], K[:, :hw], V[:, :hw], uv, valid, [(0, hw, oracle.crc_oracle.SEG_WINDOW, 0)],
                             h, w, F, 2.0, 1.0)[0]
    np.testing.assert_allclose(O[:, :hw], first, rtol=1e-13, atol=1e-13)
    full = oracle.attention(Q, K[:, :Nc], V[:, :Nc], uv, valid, cur, h, w, F, 2.0, 1.0)[0]
    np.testing.assert_array_equal(O[:, (F - 1) * hw:], full[:, (F - 1) * hw:])
    assert np.abs(O - full).max() > 1e-3  # the mask does change the earlier frames
