"""The C ABI library loads and exports every entry point include/crc.h declares,
and the ctypes mirror has the C layout.  No compute call is made (no GPU here)."""

import ctypes as C
import os
import re
import shutil
import subprocess
import tempfile

import pytest

from paper_2607_21848_gb300 import _abi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "crc.h")


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\*?\s+\*?(crc_\w+)\s*\(", text, re.M)))


@pytest.fixture(scope="module")
def lib():
    from paper_2607_21848_gb300 import build
    build.build()
    return _abi.load()


def test_header_declares_the_four_path_calls():
    names = _declared()
    for n in ("crc_retrieve", "crc_correspond", "crc_biased_attention", "crc_cache_update"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    names = _declared()
    assert names
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(_abi.EXPORTED)
    out = subprocess.run(["nm", "-D", "--defined-only", _abi.lib_path()], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (crc_\w+)", out))
    assert set(names) <= exported


def test_version_and_status_strings(lib):
    assert "sm_103a" in lib.crc_version().decode()
    for st in range(7):
        assert lib.crc_status_string(st).decode()


_LAYOUT_C = r"""
#include <stdio.h>
#include <stddef.h>
#include "crc.h"
#define P(T) printf(#T " %zu\n", sizeof(T));
#define O(T, f) printf(#T "." #f " %zu\n", offsetof(T, f));
int main(void) {
  P(crc_frame) P(crc_shape) P(crc_tensor) P(crc_segment) P(crc_cache) P(crc_bank) P(crc_retrieval) P(crc_rope)
  P(crc_step) P(crc_step_plan) O(crc_step, seg_length) O(crc_step, frames) O(crc_step_plan, bank)
  O(crc_step_plan, cache) O(crc_step_plan, retrieval) O(crc_step_plan, rope) O(crc_step_plan, eps)
  O(crc_step_plan, attn_flags) O(crc_step_plan, q) O(crc_step_plan, o) O(crc_step_plan, d_status)
  O(crc_step_plan, workspace_bytes)
  O(crc_cache, v) O(crc_cache, n_keys) O(crc_cache, seg) O(crc_bank, frames) O(crc_bank, kv) O(crc_bank, slab_chunk)
  O(crc_retrieval, delta) O(crc_retrieval, ext_min) O(crc_retrieval, exclude_sink) O(crc_shape, dtype)
  O(crc_tensor, stride_head) O(crc_rope, frame_pos0) O(crc_rope, theta)
  return 0;
}
"""


def test_ctypes_layout_matches_header():
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    with tempfile.TemporaryDirectory() as td:
        src = os.path.join(td, "layout.c")
        exe = os.path.join(td, "layout")
        open(src, "w").write(_LAYOUT_C)
        r = subprocess.run([gcc, "-I", os.path.join(ROOT, "include"), "-I", "/usr/local/cuda/include", src, "-o", exe],
                           capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
        got = dict(line.rsplit(" ", 1) for line in subprocess.run([exe], capture_output=True, text=True).stdout.split("\n")
                   if line)
    ct = {
        "crc_frame": C.sizeof(_abi.crc_frame), "crc_shape": C.sizeof(_abi.crc_shape),
        "crc_tensor": C.sizeof(_abi.crc_tensor), "crc_segment": C.sizeof(_abi.crc_segment),
        "crc_cache": C.sizeof(_abi.crc_cache), "crc_bank": C.sizeof(_abi.crc_bank),
        "crc_retrieval": C.sizeof(_abi.crc_retrieval), "crc_rope": C.sizeof(_abi.crc_rope),
        "crc_step": C.sizeof(_abi.crc_step), "crc_step_plan": C.sizeof(_abi.crc_step_plan),
        "crc_step.seg_length": _abi.crc_step.seg_length.offset, "crc_step.frames": _abi.crc_step.frames.offset,
        "crc_step_plan.bank": _abi.crc_step_plan.bank.offset, "crc_step_plan.cache": _abi.crc_step_plan.cache.offset,
        "crc_step_plan.retrieval": _abi.crc_step_plan.retrieval.offset,
        "crc_step_plan.rope": _abi.crc_step_plan.rope.offset, "crc_step_plan.eps": _abi.crc_step_plan.eps.offset,
        "crc_step_plan.attn_flags": _abi.crc_step_plan.attn_flags.offset,
        "crc_step_plan.q": _abi.crc_step_plan.q.offset, "crc_step_plan.o": _abi.crc_step_plan.o.offset,
        "crc_step_plan.d_status": _abi.crc_step_plan.d_status.offset,
        "crc_step_plan.workspace_bytes": _abi.crc_step_plan.workspace_bytes.offset,
        "crc_retrieval.exclude_sink": _abi.crc_retrieval.exclude_sink.offset,
        "crc_rope.frame_pos0": _abi.crc_rope.frame_pos0.offset, "crc_rope.theta": _abi.crc_rope.theta.offset,
        "crc_cache.v": _abi.crc_cache.v.offset, "crc_cache.n_keys": _abi.crc_cache.n_keys.offset,
        "crc_cache.seg": _abi.crc_cache.seg.offset, "crc_bank.frames": _abi.crc_bank.frames.offset,
        "crc_bank.kv": _abi.crc_bank.kv.offset,
        "crc_bank.slab_chunk": _abi.crc_bank.slab_chunk.offset, "crc_retrieval.delta": _abi.crc_retrieval.delta.offset,
        "crc_retrieval.ext_min": _abi.crc_retrieval.ext_min.offset, "crc_shape.dtype": _abi.crc_shape.dtype.offset,
        "crc_tensor.stride_head": _abi.crc_tensor.stride_head.offset,
    }
    for k, v in ct.items():
        assert int(got[k]) == v, (k, got[k], v)


def test_correspond_rejects_a_bank_beyond_32_bit_depth_offsets(lib):
    """A bank whose depth array holds 2^31 or more values is rejected on the host,
    before any CUDA call: the reprojection kernel addresses it with 32-bit offsets.
    The device pointers are placeholders that nothing dereferences."""
    F, h, w = 3, 45, 80
    cap = (2**31) // (F * h * w) + 1
    shape = _abi.crc_shape(1, 1, 64, F, h, w, _abi.CRC_F32)
    fake = 1 << 20
    bank = _abi.crc_bank(cap, 1, fake, fake, fake, fake, fake)
    frames = (_abi.crc_frame * F)()
    for f in range(F):
        frames[f].K[:] = [40.0, 0.0, 39.5, 0.0, 40.0, 22.0, 0.0, 0.0, 1.0]
        frames[f].R[:] = [1.0, 0.0, 0.0, 0.0, 1.0, 0.0, 0.0, 0.0, 1.0]
    args = (C.byref(shape), frames, fake, C.byref(bank), fake, None, 1, 0.05, fake, None, fake, None)
    assert cap * F * h * w > 2**31 - 1 >= (cap - 1) * F * h * w  # one chunk past the limit
    assert lib.crc_correspond(*args) == _abi.CRC_ERR_UNSUPPORTED


def test_retrieve_rejects_a_negative_chunk_index(lib):
    """The temporal gate n - j >= delta is evaluated in 32-bit integers; n is the
    index of the current chunk and must not be negative.  Rejected on the host,
    before any CUDA call; the device pointers are placeholders."""
    F, h, w = 3, 8, 8
    shape = _abi.crc_shape(1, 1, 64, F, h, w, _abi.CRC_F32)
    fake = 1 << 20
    bank = _abi.crc_bank(4, 1, fake, fake, fake, fake, fake)
    frames = (_abi.crc_frame * F)()
    for f in range(F):
        frames[f].K[:] = [4.0, 0.0, 3.5, 0.0, 4.0, 3.5, 0.0, 0.0, 1.0]
        frames[f].R[:] = [1.0, 0.0, 0.0, 0.0, 1.0, 0.0, 0.0, 0.0, 1.0]
    params = _abi.crc_retrieval(1.0, 0.5, float("inf"), -1.0, 1, 1, -1, 0, 0)
    assert lib.crc_retrieve(C.byref(bank), 4, C.byref(shape), frames, -1, C.byref(params), None, None, fake, None,
                            fake, None, 0, None) == _abi.CRC_ERR_INVALID_ARG
