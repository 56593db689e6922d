"""crc_host_copy: SM-issued copies between page-locked host memory and device memory.

Copies are byte work, so every case is bit-exact against the source bytes: every
direction (host to device, device to host, device to device, host to host through
the GPU), sizes from one byte to 300 MB with ragged tails, interior offsets, every
block count the launch clamps, and rejections with real buffers (pageable memory,
overlap, a misaligned pointer), which must leave the destination untouched.  The
last test runs the chunk step with its inputs uploaded and its output downloaded by
crc_host_copy on a high-priority stream, as the end-to-end bench does, and compares
the output with the step run on the device-resident inputs, bit for bit.
"""

import pytest
import torch

from paper_2607_21848_gb300 import _abi, api

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    from paper_2607_21848_gb300 import build
    build.build()
    return _abi.load()


def _pattern(n, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(0, 256, (n,), dtype=torch.uint8, generator=g)


def _buffers(n, kind, seed):
    data = _pattern(n, seed)
    if kind == "host":
        return data.pin_memory()
    return data.cuda()


@pytest.mark.parametrize("src_kind,dst_kind", [("host", "dev"), ("dev", "host"), ("dev", "dev"), ("host", "host")])
@pytest.mark.parametrize("n", [1, 15, 16, 17, 4099, 1 << 20, 10_000_019])
def test_copy_is_bit_exact_in_every_direction(lib, src_kind, dst_kind, n):
    src = _buffers(n, src_kind, 1)
    dst = _buffers(n, dst_kind, 2)
    api.crc_host_copy(dst, src)
    torch.cuda.synchronize()
    assert torch.equal(dst.cpu(), src.cpu())


@pytest.mark.parametrize("blocks", [0, 1, 3, 8, 152, 4096])
def test_block_counts_give_the_same_bytes(lib, blocks):
    n = 33_554_432 + 5  # 32 MiB and a 5-byte tail
    src = _buffers(n, "host", 3)
    dst = torch.zeros(n, dtype=torch.uint8, device="cuda")
    api.crc_host_copy(dst, src, blocks=blocks)
    torch.cuda.synchronize()
    assert torch.equal(dst.cpu(), src)


def test_large_copies_both_ways(lib):
    n = 300_000_016
    src = _buffers(n, "host", 4)
    dev = torch.empty(n, dtype=torch.uint8, device="cuda")
    back = torch.empty(n, dtype=torch.uint8, pin_memory=True)
    api.crc_host_copy(dev, src)
    api.crc_host_copy(back, dev)
    torch.cuda.synchronize()
    assert torch.equal(back, src)


def test_interior_ranges_leave_the_rest_untouched(lib):
    n = 1 << 16
    src = _buffers(n, "host", 5)
    dst = torch.zeros(n, dtype=torch.uint8, device="cuda")
    lo, cnt = 4096 + 48, 20_003
    st = lib.crc_host_copy(dst.data_ptr() + lo, src.data_ptr() + 256, cnt, 0, None)
    assert st == _abi.CRC_OK
    torch.cuda.synchronize()
    got = dst.cpu()
    assert torch.equal(got[lo:lo + cnt], src[256:256 + cnt])
    assert int(got[:lo].count_nonzero()) == 0 and int(got[lo + cnt:].count_nonzero()) == 0


def test_rejections_with_real_buffers_write_nothing(lib):
    n = 1 << 16
    pinned = _buffers(n, "host", 6)
    pageable = _pattern(n, 7)  # ordinary CPU memory: the device must not be asked to read it
    dev = torch.zeros(n, dtype=torch.uint8, device="cuda")
    assert lib.crc_host_copy(dev.data_ptr(), pageable.data_ptr(), n, 0, None) == _abi.CRC_ERR_INVALID_ARG
    assert lib.crc_host_copy(pageable.data_ptr(), dev.data_ptr(), n, 0, None) == _abi.CRC_ERR_INVALID_ARG
    # overlapping device ranges
    assert lib.crc_host_copy(dev.data_ptr() + 1024, dev.data_ptr(), 4096, 0, None) == _abi.CRC_ERR_INVALID_ARG
    assert lib.crc_host_copy(dev.data_ptr(), dev.data_ptr() + 1024, 4096, 0, None) == _abi.CRC_ERR_INVALID_ARG
    # misaligned device pointer
    assert lib.crc_host_copy(dev.data_ptr() + 8, pinned.data_ptr(), 64, 0, None) == _abi.CRC_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert int(dev.count_nonzero()) == 0
    assert torch.equal(pageable, _pattern(n, 7))


def test_the_step_through_host_copies_on_a_high_priority_stream(lib):
    """Inputs (Q, the new chunk's K/V, depth) uploaded and O downloaded by crc_host_copy on a
    high-priority stream, overlapping the previous step's kernels, as the end-to-end bench runs
    it: O equals the output of the same step on the device-resident inputs, bit for bit."""
    import bench

    W = bench.setup(1, 1, "cuda:0", seed=11)
    stream = torch.cuda.current_stream()
    bench.run_step(W, stream)
    torch.cuda.synchronize()
    ref = W["o"].clone()
    names = bench.E2E_INPUTS
    host_in = {k: W[k].cpu().pin_memory() for k in names}
    for k in names:
        W[k].zero_()
    W["o"].zero_()
    copy_s = torch.cuda.Stream(priority=-1)
    copy_s.wait_stream(stream)
    for k in names:
        api.crc_host_copy(W[k], host_in[k], stream=copy_s)
    stream.wait_stream(copy_s)
    bench.run_step(W, stream)
    out = torch.empty(W["o"].shape, dtype=W["o"].dtype, pin_memory=True)
    copy_s.wait_stream(stream)
    api.crc_host_copy(out, W["o"], stream=copy_s)
    copy_s.synchronize()
    assert torch.equal(out, ref.cpu())
