"""CPU checks of the tensor-core bias expansion's error model.

The tensor-core kernel adds the Eq. 2 bias to S as a K = 16 extension of q.k whose
large terms cancel near the correspondence.  The library states a bound on the
resulting error (crc_bias_expansion_bound, 2^-24 C (w^2 + h^2) in base-2 logit
units, besides a consistent 2^-17 scale of the bias strength) and evaluates the bias
per score where that bound exceeds 2^-9.  Here a CPU model of the kernel's own
rounding steps (tests/_tc_model.py) checks that the representation of the
coefficients takes at most a quarter of that bound, leaving the rest for the tensor
core's fp32 sum; the GPU suite measures the whole error against the same bound.
"""

import math

import numpy as np
import pytest
import torch

from paper_2607_21848_gb300 import _abi
from tests import _tc_model as M


@pytest.fixture(scope="module")
def lib():
    from paper_2607_21848_gb300 import build
    build.build()
    return _abi.load()


def test_bf16_rounding_of_the_model_matches_torch():
    g = np.random.default_rng(0)
    x = np.concatenate([g.standard_normal(4096) * 10.0 ** g.uniform(-6, 6, 4096),
                        [0.0, -0.0, 1.0, 1.00390625, 1.01171875, -3.5, 65504.0, 1e-30]]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(M.bf16(x), ref)


def test_three_term_split_of_an_fp32_value_is_exact():
    g = np.random.default_rng(1)
    v = (g.standard_normal(10000) * 10.0 ** g.uniform(-4, 6, 10000)).astype(np.float32)
    np.testing.assert_array_equal(M.split3(v), v.astype(np.float64))


@pytest.mark.parametrize("lam,sigma,h,w", [(2.0, 1.0, 30, 52), (8.0, 0.5, 45, 80), (0.7, 3.0, 8, 8),
                                           (2.0, 1.0, 256, 1)])
def test_bound_is_the_stated_closed_form(lib, lam, sigma, h, w):
    C = lam * math.log2(math.e) / (2 * sigma * sigma)
    got = lib.crc_bias_expansion_bound(lam, sigma, h, w)
    assert got == pytest.approx(C * (w * w + h * h) * 2.0 ** -24, rel=1e-6)


def test_bound_is_infinite_where_the_key_terms_are_not_exact_in_bf16(lib):
    assert math.isinf(lib.crc_bias_expansion_bound(2.0, 1.0, 1, 257))      # 2 x' = 256 needs 9 bits
    assert math.isinf(lib.crc_bias_expansion_bound(2.0, 1.0, 200, 200))    # 4 q = 199^2 + 199^2 >= 2^16
    assert not math.isinf(lib.crc_bias_expansion_bound(2.0, 1.0, 90, 160))


def test_the_configurations_bias_runs_on_the_tensor_core(lib):
    # lambda = 2, sigma = 1 on the Wan-1.3B (30 x 52) and the 14B-class (45 x 80) grids: within 2^-9
    assert lib.crc_bias_expansion_bound(2.0, 1.0, 30, 52) <= 2.0 ** -9
    assert lib.crc_bias_expansion_bound(2.0, 1.0, 45, 80) <= 2.0 ** -9
    assert lib.crc_bias_expansion_bound(8.0, 0.5, 45, 80) > 2.0 ** -9    # the steep setting: per score


@pytest.mark.parametrize("h,w", [(12, 16), (30, 52), (45, 80), (90, 160), (8, 256)])
@pytest.mark.parametrize("lam,sigma", [(2.0, 1.0), (8.0, 0.5), (32.0, 0.5)])
def test_modelled_coefficient_error_is_within_a_quarter_of_the_bound(lib, h, w, lam, sigma):
    """Correspondences anywhere on the grid (corners included) against every key cell
    whose bias is above -64 (base 2): the expansion's terms, as the kernel rounds them,
    summed exactly, differ from the bias at the applied strength A' by at most a quarter
    of the stated bound, and A' differs from the exact strength by at most 2^-17."""
    g = np.random.default_rng(h * 1000 + w)
    N = 600
    cx, cy = g.integers(0, w, N), g.integers(0, h, N)
    cx[:4], cy[:4] = [0, w - 1, 0, w - 1], [0, 0, h - 1, h - 1]
    ux = (cx + g.uniform(-0.5, 0.5, N)).astype(np.float32)
    uy = (cy + g.uniform(-0.5, 0.5, N)).astype(np.float32)
    X, Y = np.meshgrid(np.arange(w), np.arange(h))
    xk, yk = X.ravel(), Y.ravel()
    sc = float(M.kernel_constants(lam, sigma)[0])
    rep = M.expansion_terms(ux, uy, xk, yk, lam, sigma, h, w)
    strength = M.strength(lam, sigma)
    assert abs(strength - 1.0) <= 2.0 ** -17
    ex = M.exact_bias_raw(ux, uy, xk, yk, lam, sigma) * strength
    live = ex * sc > -64.0
    err = (np.abs(rep - ex) * sc)[live].max()
    bound = lib.crc_bias_expansion_bound(lam, sigma, h, w)
    assert err <= 0.25 * bound, (err, bound)


def test_expansion_is_exact_where_every_coefficient_is():
    """A head dimension of 2 and lambda = sqrt(2), sigma = 1 make the strength A' exactly -1;
    with correspondences on half-integer points every coefficient then has a few
    significant bits, its bf16 terms carry it exactly, and the expansion must equal the
    bias exactly: a wrong sign, a missing factor or a transposed term shows here."""
    lam, sigma, h, w, d = math.sqrt(2.0), 1.0, 12, 16, 2
    sc, coef, inv_sc = M.kernel_constants(lam, sigma, d)
    assert float(np.float32(coef * inv_sc)) == -1.0
    ux = np.array([0.5, 3.5, 15.5, 7.0, 8.0, 0.0], np.float32)  # x' = ux - 7.5
    uy = np.array([5.5, 0.5, 11.5, 5.0, 6.0, 0.0], np.float32)  # y' = uy - 5.5
    X, Y = np.meshgrid(np.arange(w), np.arange(h))
    rep = M.expansion_terms(ux, uy, X.ravel(), Y.ravel(), lam, sigma, h, w, d=d)
    d2 = (X.ravel()[None] - ux[:, None].astype(np.float64)) ** 2 + (Y.ravel()[None] - uy[:, None].astype(np.float64)) ** 2
    np.testing.assert_array_equal(rep, -d2)


def test_kernel_tiles_cut_segments_and_retrieved_frames():
    segs = [(0, 4680, 0, 0), (4680, 4680, 1, 0), (9360, 9360, 2, 0)]
    tiles = M.kernel_tiles(segs, 30, 52, 3)
    # sink: 37 tiles (36 full + 72 keys); retrieved: 3 frames x 13 tiles (12 full + 24 keys); window: 74 tiles
    assert len(tiles) == 37 + 39 + 74
    ret = [t for t in tiles if t[2] >= 0]
    assert all(t[4] == -1 for t in tiles)  # no current-chunk segment here
    assert [t[2] for t in ret] == [0] * 13 + [1] * 13 + [2] * 13
    assert ret[12][1] == 1560 - 12 * 128 and ret[13][0] == 4680 + 1560 and ret[13][3] == 0
    assert sum(t[1] for t in tiles) == 4680 + 4680 + 9360
