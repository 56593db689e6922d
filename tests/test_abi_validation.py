"""Host-side validation of every entry point, on the CPU, through the C ABI.

Each call below carries exactly one bad argument and must return that argument's
documented status code.  The device pointers are placeholders that nothing
dereferences: every check runs on the host before the first CUDA call, and on a
machine without a GPU any call that got as far as CUDA would return
CRC_ERR_CUDA instead.  (The GPU suite repeats these checks with real buffers and
also checks that nothing was written.)"""

import ctypes as C
import math

import pytest

from paper_2607_21848_gb300 import _abi

OK, INVALID, SHAPE, UNSUPPORTED = _abi.CRC_OK, _abi.CRC_ERR_INVALID_ARG, _abi.CRC_ERR_SHAPE, _abi.CRC_ERR_UNSUPPORTED
F, h, w, L, H, d = 3, 8, 16, 2, 2, 128
NC = F * h * w


def _ptr(i: int) -> int:
    return 0x10000000 + i * 0x01000000  # 16 MiB apart, 256-byte aligned, never dereferenced


@pytest.fixture(scope="module")
def lib():
    from paper_2607_21848_gb300 import build
    build.build()
    return _abi.load()


def _shape(**over):
    v = dict(L=L, H=H, d=d, F=F, h=h, w=w, dtype=_abi.CRC_BF16)
    v.update(over)
    return _abi.crc_shape(v["L"], v["H"], v["d"], v["F"], v["h"], v["w"], v["dtype"])


def _frames(n=F, **bad):
    fr = (_abi.crc_frame * n)()
    for f in range(n):
        fr[f].K[:] = [8.0, 0.0, 7.5, 0.0, 8.0, 3.5, 0.0, 0.0, 1.0]
        fr[f].R[:] = [1.0, 0.0, 0.0, 0.0, 1.0, 0.0, 0.0, 0.0, 1.0]
        fr[f].c[:] = [0.0, 1.6, 0.1 * f]
    for key, (e, val) in bad.items():
        getattr(fr[0], key)[e] = val
    return fr


def _bank(**over):
    v = dict(capacity=8, num_slabs=4, frames=_ptr(1), centre=_ptr(2), view=_ptr(3), depth=_ptr(4), kv=_ptr(5),
             slab_chunk=None)
    v.update(over)
    return _abi.crc_bank(v["capacity"], v["num_slabs"], v["frames"], v["centre"], v["view"], v["depth"], v["kv"],
                         v["slab_chunk"])


def _segments(k=1, window=2):
    segs = [(0, NC, _abi.CRC_SEG_SINK, 0)] + [((1 + r) * NC, NC, _abi.CRC_SEG_RETRIEVED, r) for r in range(k)] + \
           [((1 + k + q) * NC, NC, _abi.CRC_SEG_WINDOW, q) for q in range(window)]
    return segs, (1 + k + window) * NC


def _cache(segs=None, n_keys=None, k_data=None, hd=d):
    if segs is None:
        segs, n_keys = _segments()
    c = _abi.crc_cache()
    st_tok = H * hd
    c.k = _abi.crc_tensor(_ptr(6) if k_data is None else k_data, n_keys * st_tok, st_tok, hd)
    c.v = _abi.crc_tensor(_ptr(7), n_keys * st_tok, st_tok, hd)
    c.n_keys = n_keys
    c.nseg = len(segs)
    for i, s in enumerate(segs):
        c.seg[i] = _abi.crc_segment(*s)
    return c


def _params(E=1.0, w_v=0.5, tau_c=math.inf, cos_tau_v=-1.0, delta=1, k=1):
    return _abi.crc_retrieval(E, w_v, tau_c, cos_tau_v, delta, k, -1, 0, 0)


# ---- crc_bank_insert_poses ---------------------------------------------------------------------
@pytest.mark.parametrize("over, status", [
    (dict(L=0), INVALID), (dict(F=5), INVALID), (dict(h=0), INVALID),
    (dict(d=60), UNSUPPORTED), (dict(dtype=7), UNSUPPORTED), (dict(h=4096, w=4096), SHAPE),
])
def test_insert_poses_rejects_bad_shapes(lib, over, status):
    sh, b = _shape(**over), _bank()
    assert lib.crc_bank_insert_poses(C.byref(b), C.byref(sh), 0, 1, _frames(max(1, min(sh.F, 4))), None) == status


@pytest.mark.parametrize("bank_over, first, count, bad, status", [
    (dict(capacity=0), 0, 1, {}, INVALID),
    (dict(frames=None), 0, 1, {}, INVALID),
    ({}, 8, 1, {}, INVALID),                      # first + count > capacity
    ({}, 0, -1, {}, INVALID),
    ({}, -1, 1, {}, INVALID),
    ({}, 0, 1, dict(K=(0, math.nan)), INVALID),   # non-finite intrinsics
    ({}, 0, 1, dict(K=(8, 2.0)), INVALID),        # K's last row must be (0, 0, 1)
    ({}, 0, 1, dict(c=(1, math.inf)), INVALID),   # non-finite centre
])
def test_insert_poses_rejects_bad_arguments(lib, bank_over, first, count, bad, status):
    sh, b = _shape(), _bank(**bank_over)
    assert lib.crc_bank_insert_poses(C.byref(b), C.byref(sh), first, count, _frames(**bad), None) == status


def test_insert_poses_of_nothing_is_a_no_op(lib):
    sh, b = _shape(), _bank()
    assert lib.crc_bank_insert_poses(C.byref(b), C.byref(sh), 3, 0, None, None) == OK


# ---- crc_cache_update --------------------------------------------------------------------------
@pytest.mark.parametrize("case, status", [
    ("chunk_past_capacity", INVALID), ("negative_chunk", INVALID), ("k_without_v", INVALID),
    ("no_depth", INVALID), ("bad_frames", INVALID), ("misaligned_k", UNSUPPORTED),
    ("window_past_cache", SHAPE), ("no_kv_pool", INVALID),
])
def test_cache_update_rejections(lib, case, status):
    sh, b, c = _shape(), _bank(), _cache()
    chunk, fr, depth, dk, dv, woff = 1, _frames(), _ptr(8), _ptr(9), _ptr(10), 3 * NC
    if case == "chunk_past_capacity":
        chunk = 8
    elif case == "negative_chunk":
        chunk = -1
    elif case == "k_without_v":
        dv = None
    elif case == "no_depth":
        depth = None
    elif case == "bad_frames":
        fr = _frames(K=(6, 0.5))
    elif case == "misaligned_k":
        dk = _ptr(9) + 2
    elif case == "window_past_cache":
        woff = c.n_keys - NC + 1
    elif case == "no_kv_pool":
        b = _bank(kv=None)
    assert lib.crc_cache_update(C.byref(b), C.byref(sh), chunk, fr, depth, dk, dv, C.byref(c), woff, None) == status


# ---- crc_retrieve and crc_gather ---------------------------------------------------------------
@pytest.mark.parametrize("params", [_params(E=0.0), _params(E=-1.0), _params(E=math.inf), _params(k=0),
                                    _params(k=_abi.CRC_MAX_K + 1), _params(w_v=math.nan), _params(w_v=math.inf),
                                    _params(tau_c=math.nan), _params(cos_tau_v=math.nan)])
def test_retrieve_rejects_bad_parameters(lib, params):
    sh, b, c = _shape(), _bank(), _cache()
    assert lib.crc_retrieve(C.byref(b), 8, C.byref(sh), _frames(), 5, C.byref(params), C.byref(c), None, _ptr(11),
                            None, _ptr(12), None, 0, None) == INVALID


def test_retrieve_rejects_bad_counts_and_outputs(lib):
    sh, b, c, p = _shape(), _bank(), _cache(), _params()
    call = lambda count, n=5, idx=_ptr(11), cnt=_ptr(12): lib.crc_retrieve(  # noqa: E731
        C.byref(b), count, C.byref(sh), _frames(), n, C.byref(p), C.byref(c), None, idx, None, cnt, None, 0, None)
    assert call(9) == INVALID          # bank_count > capacity
    assert call(-1) == INVALID
    assert call(8, idx=None) == INVALID
    assert call(8, cnt=None) == INVALID


def test_retrieve_workspace_size_and_rejections(lib):
    size = lib.crc_retrieve_workspace_size
    assert size(512, 8) == 0 and size(0, 1) == 0          # one block: no workspace
    assert size(513, 1) > 0                                  # two blocks meet in the workspace
    assert size(100000, 3) <= size(100000, 8) <= size(10 ** 9, 8) < 300 * 1024
    assert size(2000, 0) == 0 and size(2000, _abi.CRC_MAX_K + 1) == 0 and size(-1, 1) == 0
    sh, c, p = _shape(), _cache(), _params(k=3)
    b = _bank(capacity=4096)
    need = size(4096, 3)
    call = lambda ws, nbytes: lib.crc_retrieve(  # noqa: E731
        C.byref(b), 4096, C.byref(sh), _frames(), 4096, C.byref(p), C.byref(c), None, _ptr(11), None, _ptr(12), ws,
        nbytes, None)
    assert call(None, 0) == INVALID                  # a bank of 4096 needs a workspace
    assert call(_ptr(20), need - 16) == INVALID      # too short
    assert call(_ptr(20) + 8, need) == INVALID       # not 16-byte aligned


def test_bank_slab_owner_needs_the_slab_pool(lib):
    # an owner array describes the K/V slabs: without a pool the bank is rejected
    sh, c, p = _shape(), _cache(), _params()
    b = _bank(kv=None, slab_chunk=_ptr(21))
    assert lib.crc_retrieve(C.byref(b), 8, C.byref(sh), _frames(), 5, C.byref(p), None, None, _ptr(11), None,
                            _ptr(12), None, 0, None) == INVALID


def test_retrieve_and_gather_reject_two_segments_for_one_slot(lib):
    sh, b, p = _shape(), _bank(), _params()
    dup = _cache([(0, NC, _abi.CRC_SEG_RETRIEVED, 0), (NC, NC, _abi.CRC_SEG_RETRIEVED, 0)], 2 * NC)
    assert lib.crc_retrieve(C.byref(b), 8, C.byref(sh), _frames(), 5, C.byref(p), C.byref(dup), None, _ptr(11), None,
                            _ptr(12), None, 0, None) == SHAPE
    assert lib.crc_gather(C.byref(sh), _ptr(5), 4, _ptr(11), 1, C.byref(dup), None, None) == SHAPE


@pytest.mark.parametrize("rope, status", [
    (_abi.crc_rope(0, _abi.CRC_MAX_ROPE_PAIRS + 1, 1, 0, 3, 0, 1e4), INVALID),  # too many pairs
    (_abi.crc_rope(100, 16, 1, 0, 3, 0, 1e4), INVALID),                          # channel0 + 2 pairs > d
    (_abi.crc_rope(0, 8, 1, 0, 3, 0, 0.0), INVALID),                             # theta must be > 0
    (_abi.crc_rope(0, 8, 2, 0, 3, 0, 1e4), INVALID),                             # interleaved is 0 or 1
    (_abi.crc_rope(1, 8, 1, 0, 3, 0, 1e4), UNSUPPORTED),                         # odd first channel, interleaved
    (_abi.crc_rope(4, 8, 0, 0, 3, 0, 1e4), UNSUPPORTED),                         # half-split off a 16-byte vector
    (_abi.crc_rope(0, 12, 0, 0, 3, 0, 1e4), UNSUPPORTED),
])
def test_gather_rejects_bad_rope_layouts(lib, rope, status):
    sh, c = _shape(), _cache()
    assert lib.crc_gather(C.byref(sh), _ptr(5), 4, _ptr(11), 1, C.byref(c), C.byref(rope), None) == status


def test_gather_rejects_bad_arguments(lib):
    sh, c = _shape(), _cache()
    g = lambda pool=_ptr(5), slabs=4, idx=_ptr(11), k=1, cache=C.byref(c): lib.crc_gather(  # noqa: E731
        C.byref(sh), pool, slabs, idx, k, cache, None, None)
    assert g(k=0) == INVALID
    assert g(k=_abi.CRC_MAX_K + 1) == INVALID
    assert g(idx=None) == INVALID
    assert g(cache=None) == INVALID
    assert g(pool=None) == INVALID
    assert g(slabs=0) == INVALID
    assert g(pool=_ptr(5) + 8) == UNSUPPORTED
    bad_stride = _cache()
    bad_stride.v.stride_token += 8  # K and V must share strides
    assert g(cache=C.byref(bad_stride)) == SHAPE


# ---- crc_correspond ----------------------------------------------------------------------------
@pytest.mark.parametrize("k, eps, status", [
    (0, 0.05, INVALID), (_abi.CRC_MAX_K + 1, 0.05, INVALID), (1, -0.1, INVALID), (1, math.nan, INVALID),
])
def test_correspond_rejects_bad_parameters(lib, k, eps, status):
    sh, b = _shape(), _bank()
    assert lib.crc_correspond(C.byref(sh), _frames(), _ptr(8), C.byref(b), _ptr(11), None, k, eps, _ptr(13), None,
                              _ptr(14), None) == status


def test_correspond_rejects_missing_and_misaligned_outputs(lib):
    sh, b = _shape(), _bank()
    call = lambda depth=_ptr(8), idx=_ptr(11), uv=_ptr(13), valid=_ptr(14), fr=None: lib.crc_correspond(  # noqa: E731
        C.byref(sh), _frames() if fr is None else fr, depth, C.byref(b), idx, None, 1, 0.05, uv, None, valid, None)
    assert call(depth=None) == INVALID
    assert call(idx=None) == INVALID
    assert call(uv=None) == INVALID
    assert call(valid=None) == INVALID
    assert call(fr=_frames(R=(0, math.nan))) == INVALID
    assert call(uv=_ptr(13) + 4) == UNSUPPORTED  # float2 stores need 8-byte alignment


# ---- crc_biased_attention ----------------------------------------------------------------------
def _attend(lib, cache=None, n_q=NC, k=1, lam=2.0, sigma=1.0, flags=0, uv=_ptr(13), valid=_ptr(14), sh=None,
            q_stride_head=None, hd=d):
    sh = _shape() if sh is None else sh
    q_stride_head = hd if q_stride_head is None else q_stride_head
    c = _cache(hd=hd) if cache is None else cache
    q = _abi.crc_tensor(_ptr(15), n_q * H * hd, H * hd, q_stride_head)
    o = _abi.crc_tensor(_ptr(16), n_q * H * hd, H * hd, hd)
    return lib.crc_biased_attention(C.byref(sh), q, C.byref(c), o, None, n_q, uv, valid, k, None, lam, sigma, flags,
                                    None, None)


def test_attention_rejects_bad_parameters(lib):
    assert _attend(lib, n_q=NC - 8) == SHAPE            # n_q must be N_c
    assert _attend(lib, lam=-1.0) == INVALID
    assert _attend(lib, lam=math.nan) == INVALID
    assert _attend(lib, sigma=0.0) == INVALID
    assert _attend(lib, sigma=math.inf) == INVALID
    assert _attend(lib, k=-1) == INVALID
    assert _attend(lib, k=_abi.CRC_MAX_K + 1) == INVALID
    assert _attend(lib, flags=32) == INVALID            # unknown flag bit
    assert _attend(lib, uv=None) == INVALID             # retrieved segments need correspondences
    assert _attend(lib, valid=None) == INVALID
    assert _attend(lib, k=0) == SHAPE                   # a retrieved segment's slot must be < k
    assert _attend(lib, q_stride_head=d - 8) == SHAPE   # heads of q overlap
    assert _attend(lib, uv=_ptr(13) + 4) == UNSUPPORTED  # correspondences are read as float2


def test_attention_rejects_bad_segment_tables(lib):
    overlap = _cache([(0, 2 * NC, _abi.CRC_SEG_SINK, 0), (NC, NC, _abi.CRC_SEG_WINDOW, 0)], 3 * NC)
    assert _attend(lib, cache=overlap) == SHAPE
    assert _attend(lib, cache=_cache([(0, NC, 7, 0)], NC)) == INVALID          # unknown kind
    assert _attend(lib, cache=_cache([(0, NC - 1, _abi.CRC_SEG_RETRIEVED, 0)], NC)) == SHAPE  # not a whole chunk
    assert _attend(lib, cache=_cache([(NC, NC, _abi.CRC_SEG_SINK, 0)], NC)) == SHAPE  # past the cache
    too_many = _cache([(i, 1, _abi.CRC_SEG_WINDOW, 0) for i in range(_abi.CRC_MAX_SEGMENTS)], NC)
    too_many.nseg = _abi.CRC_MAX_SEGMENTS + 1
    assert _attend(lib, cache=too_many) == SHAPE
    misaligned = _cache(k_data=_ptr(6) + 8)
    assert _attend(lib, cache=misaligned) == UNSUPPORTED
    # the current chunk's segment is a whole chunk (cut per frame), or empty
    assert _attend(lib, cache=_cache([(0, NC - 1, _abi.CRC_SEG_CURRENT, 0)], NC)) == SHAPE


def test_attention_limits_of_the_tensor_core_kernel(lib):
    # bf16 with d = 64 is not a tensor-core shape (the SIMT flag takes it)
    assert _attend(lib, sh=_shape(d=64), hd=64) == UNSUPPORTED
    # 640 KV tiles of 128 keys is the kernel's limit: 641 window tiles are one too many
    n_keys = 641 * 128
    segs = [(0, n_keys, _abi.CRC_SEG_WINDOW, 0)]
    assert _attend(lib, cache=_cache(segs, n_keys), k=0, uv=None, valid=None) == UNSUPPORTED


@pytest.mark.parametrize("dst, src, nbytes, blocks, status", [
    (_ptr(1), _ptr(2), 0, 0, OK),                  # nothing to copy: nothing enqueued
    (None, _ptr(2), 64, 0, INVALID),
    (_ptr(1), None, 64, 0, INVALID),
    (_ptr(1), _ptr(2), 64, -1, INVALID),
    (_ptr(1), _ptr(2), 64, 4097, INVALID),
    (_ptr(1) + 8, _ptr(2), 64, 0, UNSUPPORTED),    # 16-byte alignment of both pointers
    (_ptr(1), _ptr(2) + 4, 64, 0, UNSUPPORTED),
])
def test_host_copy_rejections_before_any_cuda_call(lib, dst, src, nbytes, blocks, status):
    assert lib.crc_host_copy(dst, src, nbytes, blocks, None) == status
