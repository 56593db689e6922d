"""A CPU model of the tensor-core attention kernel's own arithmetic (test infrastructure).

This is not the oracle: the oracle states Eq. 2 exactly; this module restates the
rounding steps the kernel takes, in numpy float32 / bfloat16 emulation, so that the
tests can tell which part of the kernel's deviation from the oracle each step
explains.  It shares no code with the CUDA library.

  expansion_terms    the K = 16 bias extension of q.k: A rounded to two bf16 terms (A'),
                     the query-side coefficients -2A' ux', -2A' uy', A'(ux'^2 + uy'^2)
                     formed in double-fp32 and split into 4, 4 and 3 bf16 terms, the
                     key-side q_k (two bf16 terms), x', y'; their products summed
                     exactly (fp64).
  attention_model    the softmax protocol per 128-key tile (tile cut per segment and,
                     in retrieved segments, per frame; the stale row max refreshed
                     only when it grows by more than 2^8; P = 2^(s sc - m) rounded to
                     bf16 for P V; the row sum from the fp32 P; O scaled once at the
                     end and rounded to bf16), with S taken as the fp32 rounding of
                     the exact q.k plus the modelled bias.
"""

from __future__ import annotations

import math

import numpy as np

LOG2E = 1.4426950408889634
f32 = np.float32


def bf16(x):
    """Round float32 values to bfloat16 (nearest even), returned as float32 of x's shape."""
    x = np.asarray(x, dtype=np.float32)
    a = np.ascontiguousarray(x).reshape(-1)
    u = a.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32)
    return np.where(np.isfinite(a), out, a).reshape(x.shape)


def split3(v):
    """v (float32) ~= hi + mid + lo in bf16, each term rounded from the remainder."""
    v = np.asarray(v, dtype=np.float32)
    hi = bf16(v)
    r1 = (v - hi).astype(np.float32)
    mid = bf16(r1)
    r2 = (r1 - mid).astype(np.float32)
    lo = bf16(r2)
    return hi.astype(np.float64) + mid.astype(np.float64) + lo.astype(np.float64)


def two_prod(a, b):
    """a b = p + e with p the fp32 product and e its exact error (both float32)."""
    a = np.asarray(a, np.float32)
    b = np.asarray(b, np.float32)
    p = (a * b).astype(np.float32)
    e = (a.astype(np.float64) * b.astype(np.float64) - p.astype(np.float64)).astype(np.float32)
    return p, e


def split_df(hi, lo, n):
    """hi + lo as n bf16 terms, each the nearest bf16 to what remains; lo joins the
    remainder after the first term (fp32 arithmetic).  Returns the sum of the terms (float64)."""
    r = np.asarray(hi, np.float32)
    tot = np.zeros(r.shape)
    for i in range(n):
        t = bf16(r)
        tot = tot + t.astype(np.float64)
        r = (r - t).astype(np.float32)
        if i == 0:
            r = (r + np.asarray(lo, np.float32)).astype(np.float32)
    return tot


def fma32(a, b, c):
    """fp32 fused multiply-add (one rounding), via float64."""
    return (np.asarray(a, np.float64) * np.asarray(b, np.float64) + np.asarray(c, np.float64)).astype(np.float32)


def kernel_constants(lam: float, sigma: float, d: int = 128):
    """The fp32 constants the launch computes in fp64 and the kernel derives from them."""
    sc = f32(LOG2E / math.sqrt(d))
    coef = f32(-lam * LOG2E / (2.0 * sigma * sigma))
    inv_sc = f32(f32(1.0) / sc)
    return sc, coef, inv_sc


def expansion_terms(ux, uy, xk, yk, lam, sigma, h, w, d: int = 128):
    """The raw-unit bias the K = 16 extension contributes for correspondences (ux, uy)
    [N] against key cells (xk, yk) [M], with every product exact: [N, M] float64.
    Modelled: A rounded to two bf16 terms (A'); -2 A' ux', -2 A' uy' and A' (ux'^2 + uy'^2)
    formed in double-fp32 and split into 4, 4 and 3 bf16 terms; q_k in two terms.  The
    tensor core's own summation is not."""
    sc, coef, inv_sc = kernel_constants(lam, sigma, d)
    xc, yc = f32(0.5) * f32(w - 1), f32(0.5) * f32(h - 1)
    A = f32(coef * inv_sc)
    ah = bf16(A)
    al = bf16(np.float32(A - ah))
    ux_ = (np.asarray(ux, np.float32) - xc).astype(np.float32)
    uy_ = (np.asarray(uy, np.float32) - yc).astype(np.float32)
    p, e = two_prod(np.full(ux_.shape, ah, np.float32), ux_)
    c1 = split_df((f32(-2.0) * p).astype(np.float32), (f32(-2.0) * fma32(al, ux_, e)).astype(np.float32), 4)
    p, e = two_prod(np.full(uy_.shape, ah, np.float32), uy_)
    c2 = split_df((f32(-2.0) * p).astype(np.float32), (f32(-2.0) * fma32(al, uy_, e)).astype(np.float32), 4)
    sx, ex = two_prod(ux_, ux_)
    sy, ey = two_prod(uy_, uy_)
    sq = (sx + sy).astype(np.float32)  # two_sum: the exact error of the fp32 sum
    es = (sx.astype(np.float64) + sy.astype(np.float64) - sq.astype(np.float64)).astype(np.float32)
    sl = ((ex + ey).astype(np.float32) + es).astype(np.float32)
    p, e = two_prod(np.full(sq.shape, ah, np.float32), sq)
    c3 = split_df(p, fma32(ah, sl, fma32(al, sq, e)), 3)
    xr = (np.asarray(xk, np.float64) - float(xc))
    yr = (np.asarray(yk, np.float64) - float(yc))
    q = xr * xr + yr * yr
    qh = bf16(q.astype(np.float32)).astype(np.float64)
    ql = bf16((q - qh).astype(np.float32)).astype(np.float64)
    xb = bf16(xr.astype(np.float32)).astype(np.float64)
    yb = bf16(yr.astype(np.float32)).astype(np.float64)
    a = float(ah) + float(al)
    return (a * (qh + ql)[None] + c1[:, None] * xb[None] + c2[:, None] * yb[None] + c3[:, None])


def strength(lam, sigma, d: int = 128):
    """The bias strength the expansion applies, A' (two bf16 terms of A), over the exact
    lambda sqrt(d) / (2 sigma^2): the consistent scale of the tensor core's bias."""
    sc, coef, inv_sc = kernel_constants(lam, sigma, d)
    A = f32(coef * inv_sc)
    ah = bf16(A)
    return (float(ah) + float(bf16(np.float32(A - ah)))) / (-lam * math.sqrt(d) / (2.0 * sigma * sigma))


def exact_bias_raw(ux, uy, xk, yk, lam, sigma, d: int = 128):
    """Eq. 2's lambda B in the kernel's raw score units (lambda sqrt(d) B), float64."""
    d2 = (np.asarray(xk, np.float64)[None] - np.asarray(ux, np.float64)[:, None]) ** 2 + \
         (np.asarray(yk, np.float64)[None] - np.asarray(uy, np.float64)[:, None]) ** 2
    return -lam * math.sqrt(d) * d2 / (2.0 * sigma * sigma)


def kernel_tiles(segments, h, w, F, slot_chunks=None, BN=128, frame_causal=False):
    """The kernel's KV tiles: (first key, active keys, source frame or -1, index of the
    first key inside its frame, current-chunk frame or -1), in segment order, retrieved
    segments (and, in the frame-causal mode, the current chunk's) cut per frame."""
    tiles = []
    hw = h * w
    for off, length, kind, slot in segments:
        if length <= 0:
            continue
        ret, cur = kind == 1, kind == 3 and frame_causal
        if ret and slot_chunks is not None and slot_chunks[slot] < 0:
            continue
        for rr in range(F if (ret or cur) else 1):
            start = off + rr * hw if (ret or cur) else off
            rlen = hw if (ret or cur) else length
            for t in range((rlen + BN - 1) // BN):
                tiles.append((start + t * BN, min(BN, rlen - t * BN), slot * F + rr if ret else -1, t * BN,
                              rr if cur else -1))
    return tiles


def attention_model(Q, Kc, Vc, uv, valid, segments, h, w, F, lam, sigma, slot_chunks=None, bias="tensor",
                    mask_mode="chunk"):
    """O [L, Nq, H, d] (bf16 values as float64) and LSE [L, H, Nq] following the kernel's
    rounding steps.  bias = "tensor" (the K = 16 expansion, exact products) or "direct"
    (fp32 per score, as the kernel's per-score form).  mask_mode = "frame": a row whose
    query frame precedes a current-chunk tile's frame takes no weight from that tile and
    keeps its max and sum."""
    L, Nq, H, d = Q.shape
    sc, coef, inv_sc = kernel_constants(lam, sigma, d)
    tiles = kernel_tiles(segments, h, w, F, slot_chunks, frame_causal=mask_mode == "frame")
    O = np.zeros((L, Nq, H, d))
    LSE = np.zeros((L, H, Nq))
    uv32 = np.asarray(uv, np.float32)
    for l in range(L):
        for hh in range(H):
            q = Q[l, :, hh, :].astype(np.float64)
            m = np.full(Nq, -np.inf, np.float32)
            lsum = np.zeros(Nq, np.float32)
            acc = np.zeros((Nq, d), np.float32)
            qframe = np.arange(Nq) // (h * w)
            for j, (k0, nact, s, loc0, kf) in enumerate(tiles):
                rowmask = (kf >= 0) & (kf > qframe)
                kk = Kc[l, k0:k0 + nact, hh, :].astype(np.float64)
                vv = Vc[l, k0:k0 + nact, hh, :].astype(np.float64)
                S = q @ kk.T  # exact products; fp32 rounding below
                if s >= 0 and lam != 0.0:
                    loc = loc0 + np.arange(nact)
                    xk, yk = loc % w, loc // w
                    ok = valid[:, s].astype(bool)
                    if bias == "tensor":
                        b = expansion_terms(uv32[:, s, 0], uv32[:, s, 1], xk, yk, lam, sigma, h, w, d)
                    else:
                        araw = f32(coef * inv_sc)
                        dx = (uv32[:, s, 0][:, None] - xk[None].astype(np.float32)).astype(np.float32)
                        dy = (uv32[:, s, 1][:, None] - yk[None].astype(np.float32)).astype(np.float32)
                        d2 = (dx.astype(np.float64) * dx + (dy * dy).astype(np.float32)).astype(np.float32)
                        b = (araw * d2.astype(np.float64))
                    S = S + np.where(ok[:, None], b, 0.0)
                S32 = S.astype(np.float32)
                mt = np.where(rowmask, -np.inf, (S32.max(axis=1) * sc)).astype(np.float32)
                mnew = np.maximum(m, mt)
                resc = mnew > (m + f32(8.0)).astype(np.float32)
                with np.errstate(invalid="ignore", over="ignore"):
                    factor = np.where(resc, np.exp2((m - mnew).astype(np.float64)).astype(np.float32), f32(1.0))
                m = np.where(resc, mnew, m).astype(np.float32)
                t = (S32.astype(np.float64) * float(sc) - m[:, None].astype(np.float64)).astype(np.float32)
                t[rowmask] = -np.inf
                p = np.exp2(t.astype(np.float64)).astype(np.float32)
                psum = p.astype(np.float64).sum(axis=1).astype(np.float32)
                lsum = (lsum * factor + psum).astype(np.float32)
                if j > 0:
                    acc = (acc * factor[:, None]).astype(np.float32)
                acc = (acc + (bf16(p).astype(np.float64) @ vv).astype(np.float32)).astype(np.float32)
            inv = np.where(lsum > 0, (f32(1.0) / np.where(lsum > 0, lsum, f32(1.0))).astype(np.float32), f32(0.0))
            O[l, :, hh, :] = bf16((acc * inv[:, None]).astype(np.float32)).astype(np.float64)
            with np.errstate(divide="ignore"):
                LSE[l, hh] = np.where(lsum > 0, (m.astype(np.float64) + np.log2(lsum.astype(np.float64))) * math.log(2),
                                      -np.inf)
    return O, LSE
