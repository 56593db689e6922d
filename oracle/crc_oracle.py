"""fp64 CPU oracle for the per-chunk revisit-consistency path.

TEST INFRASTRUCTURE ONLY.  This module is the plain, slow, literal statement of
what the path computes, used to check the CUDA library.  Only the test suite,
the smoke check and the benchmark's CPU-baseline / reference arm may import it;
the product path never does.  It shares no code with the CUDA library and
imports nothing from it.

Every function follows one passage of the paper ("Closing the Loop:
Training-Free Revisit Consistency for Autoregressive Generative Rendering"):

  chunk_pose        Sec. 4.2 (camera centre c_n and unit view direction v_n of a chunk)
  retrieve          Sec. 4.2, Eq. 1 (score s(j), admissible set A_n, empty-set fallback)
  fill_slots        Sec. 4.2 (an empty A_n makes the retrieved slot extend the recent window)
  gather            Sec. 4.2 (retrieved chunk reinstated into the clean cache)
  rope_reposition   Sec. 4.2 "Cache packing" (re-packed chunk moved to positions next to the window)
  reproject         Sec. 4.3, Eq. 3 (reprojection warp)
  correspond        Sec. 4.3, Eq. 3-4 and the design choices (visibility test, exact fallback)
  key_table         Sec. 4.3 design choice (ii) (which key columns carry a bias)
  attention         Sec. 4.3, Eq. 2 (biased logits, softmax, weighted sum of values)

Readings of points the paper leaves open (all listed with the design notes):
  * (c_n, v_n) of a chunk: mean of its frames' centres; the normalised sum of
    its frames' optical axes (third column of R), summed in frame order.
  * top-k for k > 1: the k admissible chunks with the smallest (s, j), ascending.
  * token (row i, col j) has grid coordinate (j, i); the landing cell of u-hat
    is (floor(x + 1/2), floor(y + 1/2)); "off-grid" = cell outside the grid.
  * Eq. 4 reads D_s at the landing cell; eps = +inf disables the test.
  * "behind the camera" = [X_s]_z <= 0; a non-finite or non-positive query
    depth is also undefined.
  * A slot that holds a window-extension chunk (not a pose retrieval) is not a
    retrieved chunk, so its correspondences are all invalid (no bias).

Each function has independent pins in tests/test_oracle.py (hand-worked
retrievals, identity pose, the pure-translation closed form, the pure-rotation
homography, the analytic-scene round trip, brute-force softmax, library SDPA).
"""

from __future__ import annotations

import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

SEG_SINK = 0
SEG_RETRIEVED = 1
SEG_WINDOW = 2
SEG_CURRENT = 3  # the window slot holding the current chunk (a window segment otherwise)


# ----------------------------------------------------------------------------
# Sec. 4.2 — chunk pose and loop-closure retrieval (Eq. 1)
# ----------------------------------------------------------------------------


def chunk_pose(R: np.ndarray, c: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Camera centre and unit viewing direction of a chunk from its F frames.

    R: [F, 3, 3] camera-to-world rotations, c: [F, 3] centres.  The centre is the
    mean of the frame centres; the view direction is the sum of the frames'
    optical axes (R[:, :, 2]) normalised to unit length.  Sums run in frame order.
    """
    F = c.shape[0]
    cs = np.array(c[0], dtype=np.float64)
    vs = np.array(R[0][:, 2], dtype=np.float64)
    for f in range(1, F):
        cs = cs + c[f]
        vs = vs + R[f][:, 2]
    centre = cs / float(F)
    norm = math.sqrt(vs[0] * vs[0] + vs[1] * vs[1] + vs[2] * vs[2])
    view = np.array([vs[0] / norm, vs[1] / norm, vs[2] / norm])
    return centre, view


def retrieval_terms(bank_c: np.ndarray, bank_v: np.ndarray, c_n: np.ndarray, v_n: np.ndarray,
                    E: float, w_v: float):
    """Eq. 1 for every bank entry j: (s(j), ||c_j - c_n||/E, v_j . v_n)."""
    dx = bank_c[:, 0] - c_n[0]
    dy = bank_c[:, 1] - c_n[1]
    dz = bank_c[:, 2] - c_n[2]
    dist = np.sqrt(dx * dx + dy * dy + dz * dz) / E
    dot = bank_v[:, 0] * v_n[0] + bank_v[:, 1] * v_n[1] + bank_v[:, 2] * v_n[2]
    s = dist + w_v * (1.0 - dot)
    return s, dist, dot


def retrieve(bank_c: np.ndarray, bank_v: np.ndarray, c_n: np.ndarray, v_n: np.ndarray, n: int,
             E: float, w_v: float, tau_c: float, cos_tau_v: float, delta: int, k: int,
             exclude_sink: bool = False, resident: Optional[np.ndarray] = None):
    """Eq. 1: score every historical chunk j, keep the admissible set A_n, and return
    the k admissible chunks closest in pose (ascending (s, j)).  With exclude_sink
    the anchor chunk j = 0 (always in the cache already) is never admissible.

    resident [B] bool (optional): chunks whose keys and values are still held.  The
    paper keeps every chunk re-encodable (Sec. 4.2); a store of bounded size can
    only reinstate the chunks it still holds, so the others are not admissible.

    Returns (idx [k] int32 padded with -1, score [k] fp64 padded with +inf, count).
    """
    B = bank_c.shape[0]
    s, dist, dot = retrieval_terms(bank_c, bank_v, c_n, v_n, E, w_v)
    j = np.arange(B)
    adm = (dist <= tau_c) & (dot >= cos_tau_v) & ((n - j) >= delta)
    if exclude_sink:
        adm &= j != 0
    if resident is not None:
        adm &= np.asarray(resident, dtype=bool)[:B]
    cand = sorted((float(s[i]), int(i)) for i in np.nonzero(adm)[0])
    count = min(k, len(cand))
    idx = np.full(k, -1, dtype=np.int32)
    score = np.full(k, np.inf)
    for r in range(count):
        score[r], idx[r] = cand[r]
    return idx, score, count


def fill_slots(idx: np.ndarray, count: int, ext_first: int, ext_min: int,
               resident: Optional[np.ndarray] = None) -> np.ndarray:
    """Chunk held by each retrieved slot.  Slots r < count hold the retrieval result;
    the rest extend the recent window with the next-older chunks ext_first,
    ext_first-1, ... while they are >= ext_min (and, given `resident`, still held),
    else stay empty (-1)."""
    k = idx.shape[0]
    out = np.array(idx, dtype=np.int32)
    for r in range(count, k):
        e = ext_first - (r - count)
        ok = ext_first >= 0 and e >= ext_min
        if ok and resident is not None:
            ok = bool(resident[e])
        out[r] = e if ok else -1
    return out


def rope_frequencies(pairs: int, theta: float) -> np.ndarray:
    """Angular frequency of each temporal rotary pair i: theta^(-i / pairs)."""
    return np.array([theta ** (-(i / pairs)) for i in range(pairs)], dtype=np.float64)


def rope_reposition(x: np.ndarray, delta: float, channel0: int, pairs: int, theta: float,
                    interleaved: bool) -> np.ndarray:
    """Sec. 4.2 "Cache packing": move keys that carry a rotary embedding at temporal
    position t to position t + delta.  Each temporal pair (x_a, x_b) is read as the
    complex number x_a + i x_b and multiplied by exp(i delta omega_i).  Pair i sits at
    channels (channel0 + 2i, channel0 + 2i + 1) when interleaved, else at
    (channel0 + i, channel0 + i + pairs).  x [..., d] is widened to fp64."""
    out = np.array(x, dtype=np.float64)
    omega = rope_frequencies(pairs, theta)
    for i in range(pairs):
        if interleaved:
            a, b = channel0 + 2 * i, channel0 + 2 * i + 1
        else:
            a, b = channel0 + i, channel0 + i + pairs
        z = (out[..., a] + 1j * out[..., b]) * np.exp(1j * (delta * omega[i]))
        out[..., a] = z.real
        out[..., b] = z.imag
    return out


def gather(pool: np.ndarray, slot_chunks: np.ndarray, num_slabs: int,
           rope: Optional[dict] = None) -> List[Optional[np.ndarray]]:
    """Reinstate chunk slot_chunks[r] (slab chunk % num_slabs of pool [P, 2, L, Nc, H, d]).

    With `rope` (keys channel0, pairs, theta, interleaved, pos_slot0, pos_stride,
    frame_pos0, F) the keys of slot r, cached at positions frame_pos0 + j F + f, are
    moved to pos_slot0 + r pos_stride + f (Sec. 4.2 "Cache packing": the retrieved
    chunk is re-packed next to the recent window).  Values carry no rotary embedding."""
    out: List[Optional[np.ndarray]] = []
    for r, j in enumerate(slot_chunks):
        if j < 0:
            out.append(None)
            continue
        slab = np.array(pool[j % num_slabs], dtype=np.float64)
        if rope is not None and rope["pairs"] > 0:
            delta = (rope["pos_slot0"] + r * rope["pos_stride"]) - (rope["frame_pos0"] + int(j) * rope["F"])
            slab[0] = rope_reposition(slab[0], delta, rope["channel0"], rope["pairs"], rope["theta"],
                                      rope["interleaved"])
        out.append(slab)
    return out


# ----------------------------------------------------------------------------
# Sec. 4.3 — reprojection warp (Eq. 3) and visibility (Eq. 4)
# ----------------------------------------------------------------------------


def reproject(u: np.ndarray, z: np.ndarray, Kt: np.ndarray, Rt: np.ndarray, ct: np.ndarray,
              Ks: np.ndarray, Rs: np.ndarray, cs: np.ndarray):
    """Eq. 3 for points u [N, 2] (grid x, y) with planar depth z [N] in the target
    camera t: X_t = z K_t^-1 u~,  X_s = R_s^T (R_t X_t + c_t - c_s),  u^ = pi(K_s X_s).

    Returns (u_hat [N, 2], X_s [N, 3])."""
    u_h = np.concatenate([u, np.ones((u.shape[0], 1))], axis=1)  # homogeneous grid coordinates
    Xt = z[:, None] * (np.linalg.inv(Kt) @ u_h.T).T
    Xs = (Rs.T @ ((Rt @ Xt.T).T + ct - cs).T).T
    q = (Ks @ Xs.T).T
    with np.errstate(divide="ignore", invalid="ignore"):
        u_hat = q[:, :2] / q[:, 2:3]
    return u_hat, Xs


def correspond(depth_t: np.ndarray, Kt: np.ndarray, Rt: np.ndarray, ct: np.ndarray,
               depth_s: np.ndarray, Ks: np.ndarray, Rs: np.ndarray, cs: np.ndarray,
               eps: float, source_ok: Optional[np.ndarray] = None, with_zs: bool = False):
    """Correspondence of every query token of the current chunk in every source frame.

    depth_t [F, h, w], Kt/Rt [F, 3, 3], ct [F, 3]: current (target) frames.
    depth_s [S, h, w], Ks/Rs [S, 3, 3], cs [S, 3]: source frames (retrieved slots x F).
    source_ok [S]: False for frames of slots that hold no pose-retrieved chunk.

    Query p = (t, i, j) = frame t, row i, col j in row-major order.  Returns
    uv [Nq, S, 2] (u-hat, fp64), cell [Nq, S] int32 (y*w + x, -1 if invalid) and
    valid [Nq, S] bool, where valid means: the query depth is finite and positive,
    u-hat is finite, the point is in front of the source camera, the landing cell
    is on the grid, and Eq. 4 holds ([X_s]_z <= (1 + eps) D_s(cell)).
    With `with_zs`, also returns [X_s]_z [Nq, S] (the point's depth in the source camera).
    """
    F, h, w = depth_t.shape
    S = depth_s.shape[0]
    Nq = F * h * w
    ii, jj = np.meshgrid(np.arange(h, dtype=np.float64), np.arange(w, dtype=np.float64), indexing="ij")
    u = np.stack([jj.ravel(), ii.ravel()], axis=1)
    uv = np.zeros((Nq, S, 2))
    cell = np.full((Nq, S), -1, dtype=np.int32)
    valid = np.zeros((Nq, S), dtype=bool)
    zs = np.zeros((Nq, S))
    for t in range(F):
        z = depth_t[t].astype(np.float64).ravel()
        rows = slice(t * h * w, (t + 1) * h * w)
        for s in range(S):
            u_hat, Xs = reproject(u, z, Kt[t], Rt[t], ct[t], Ks[s], Rs[s], cs[s])
            uv[rows, s] = u_hat
            zs[rows, s] = Xs[:, 2]
            with np.errstate(invalid="ignore"):
                cx = np.floor(u_hat[:, 0] + 0.5)
                cy = np.floor(u_hat[:, 1] + 0.5)
                ok = np.isfinite(z) & (z > 0) & np.isfinite(u_hat).all(axis=1) & (Xs[:, 2] > 0)
                ok &= (cx >= 0) & (cx < w) & (cy >= 0) & (cy < h)
            xi = np.where(ok, cx, 0).astype(np.int64)
            yi = np.where(ok, cy, 0).astype(np.int64)
            if not math.isinf(eps):
                Ds = depth_s[s].astype(np.float64)[yi, xi]
                ok &= Xs[:, 2] <= (1.0 + eps) * Ds
            if source_ok is not None and not source_ok[s]:
                ok[:] = False
            valid[rows, s] = ok
            cell[rows, s] = np.where(ok, yi * w + xi, -1)
    if with_zs:
        return uv, cell, valid, zs
    return uv, cell, valid


# ----------------------------------------------------------------------------
# Sec. 4.3 — biased attention (Eq. 2)
# ----------------------------------------------------------------------------


def key_table(segments: Sequence[Tuple[int, int, int, int]], n_keys: int, h: int, w: int, F: int,
              slot_chunks: Optional[np.ndarray] = None):
    """Per key column: active flag, source frame s (-1 when the column carries no bias)
    and grid position u_k = (x, y) within that source frame.

    Keys outside every segment, or in a retrieved slot that holds no chunk, are
    inactive (masked).  Only RETRIEVED columns get a source frame (design
    choice ii); s = slot * F + (position in slot) // (h w).
    """
    active = np.zeros(n_keys, dtype=bool)
    src = np.full(n_keys, -1, dtype=np.int64)
    ux = np.zeros(n_keys)
    uy = np.zeros(n_keys)
    for off, length, kind, slot in segments:
        if length <= 0:
            continue
        if kind == SEG_RETRIEVED and slot_chunks is not None and slot_chunks[slot] < 0:
            continue
        active[off:off + length] = True
        if kind == SEG_RETRIEVED:
            loc = np.arange(length)
            src[off:off + length] = slot * F + loc // (h * w)
            rem = loc % (h * w)
            ux[off:off + length] = rem % w
            uy[off:off + length] = rem // w
    return active, src, ux, uy


def bias_matrix(uv: np.ndarray, valid: np.ndarray, rows: np.ndarray, src: np.ndarray, ux: np.ndarray,
                uy: np.ndarray, sigma: float, form: str = "eq2") -> np.ndarray:
    """Eq. 2 bias B_s(p, k) = -||u_k - u^_s(p)||^2 / (2 sigma^2) for query rows `rows`;
    zero on columns without a source frame and for invalid correspondences.

    form = "gaussian" is the opt-in additive variant exp(-||u_k - u^_s(p)||^2 / (2 sigma^2))
    (a bonus that peaks at the correspondence) in place of Eq. 2's quadratic penalty."""
    B = np.zeros((rows.shape[0], src.shape[0]))
    for s in np.unique(src[src >= 0]):
        cols = np.nonzero(src == s)[0]
        uhx = uv[rows, s, 0].astype(np.float64)[:, None]
        uhy = uv[rows, s, 1].astype(np.float64)[:, None]
        d2 = (ux[cols][None, :] - uhx) ** 2 + (uy[cols][None, :] - uhy) ** 2
        b = -d2 / (2.0 * sigma * sigma)
        if form == "gaussian":
            b = np.exp(b)
        elif form != "eq2":
            raise ValueError(form)
        b = np.where(valid[rows, s].astype(bool)[:, None], b, 0.0)
        B[:, cols] = b
    return B


def current_key_frames(segments, n_keys: int, h: int, w: int) -> np.ndarray:
    """Per key column: the latent frame of the current chunk the key belongs to (keys of
    the CURRENT segment, position // (h w)), -1 for every other key."""
    kf = np.full(n_keys, -1, dtype=np.int64)
    for off, length, kind, _ in segments:
        if kind == SEG_CURRENT and length > 0:
            kf[off:off + length] = np.arange(length) // (h * w)
    return kf


def attention(Q: np.ndarray, Kc: np.ndarray, Vc: np.ndarray, uv: np.ndarray, valid: np.ndarray,
              segments, h: int, w: int, F: int, lam: float, sigma: float,
              slot_chunks: Optional[np.ndarray] = None, rows: Optional[np.ndarray] = None,
              layers: Optional[Sequence[int]] = None, heads: Optional[Sequence[int]] = None,
              row_block: int = 1024, bias_form: str = "eq2", mask_mode: str = "chunk"):
    """Eq. 2: O_p = sum_k softmax_k(A_pk) V_k with A_pk = q_p.k_k / sqrt(d) + lam B_s(p, k).
    bias_form selects the bias of `bias_matrix` (Eq. 2, or the opt-in additive Gaussian).

    mask_mode "chunk": every active key is visible to every query (chunks attend
    block-causally, Sec. 3, and every cached key belongs to this chunk or an earlier one).
    "frame": frame-causal inside the current chunk -- a query of latent frame t = p // (h w)
    does not see the keys of the CURRENT segment whose frame is later than t.

    Q [L, Nq, H, d], Kc/Vc [L, Nk, H, d] (values as given, widened to fp64),
    uv [Nq, S, 2], valid [Nq, S].  Softmax runs over the active keys only, in two
    passes (row max, then exp-sum).  Returns O [L', R, H', d] and the natural-log
    LSE [L', H', R] for the selected layers / heads / query rows.
    """
    L, Nq, H, d = Q.shape
    Nk = Kc.shape[1]
    rows = np.arange(Nq) if rows is None else np.asarray(rows)
    layers = list(range(L)) if layers is None else list(layers)
    heads = list(range(H)) if heads is None else list(heads)
    active, src, ux, uy = key_table(segments, Nk, h, w, F, slot_chunks)
    act = np.nonzero(active)[0]
    if mask_mode not in ("chunk", "frame"):
        raise ValueError(mask_mode)
    kframe = current_key_frames(segments, Nk, h, w)[act]
    O = np.zeros((len(layers), rows.shape[0], len(heads), d))
    lse = np.zeros((len(layers), len(heads), rows.shape[0]))
    scale = 1.0 / math.sqrt(d)
    for b0 in range(0, rows.shape[0], row_block):
        rb = rows[b0:b0 + row_block]
        lamB = lam * bias_matrix(uv, valid, rb, src[act], ux[act], uy[act], sigma, bias_form)
        for li, l in enumerate(layers):
            for hi, hh in enumerate(heads):
                q = Q[l, rb, hh, :].astype(np.float64)
                k = Kc[l, act, hh, :].astype(np.float64)
                v = Vc[l, act, hh, :].astype(np.float64)
                A = (q @ k.T) * scale + lamB
                if mask_mode == "frame":
                    qframe = rb // (h * w)
                    A = np.where(kframe[None, :] > qframe[:, None], -np.inf, A)
                m = A.max(axis=1, keepdims=True)
                e = np.exp(A - m)
                ssum = e.sum(axis=1, keepdims=True)
                O[li, b0:b0 + rb.shape[0], hi, :] = (e @ v) / ssum
                lse[li, hi, b0:b0 + rb.shape[0]] = (m + np.log(ssum))[:, 0]
    return O, lse
