"""Host-side layout of the chunk stream (no GPU): which cache region holds which chunk
at step n, which segments are live, the window-extension fallback chunk, and the
rotary positions of the re-packed retrieved slots (Sec. 4.2 "Cache layout" and
"Cache packing").  The cache contents are simulated here from the writes a step
makes (chunk n into ring slot n % W, chunk 0 into the sink) and compared with what
the stream declares."""

import pytest

from paper_2607_21848_gb300 import api
from paper_2607_21848_gb300.stream import ChunkStream, StreamConfig


def _stream(k=2, window=2, F=3, h=4, w=5, rope_pairs=0):
    cfg = StreamConfig(L=1, H=1, d=64, F=F, h=h, w=w, k=k, window=window, capacity=64, num_slabs=4, E=1.0, w_v=0.5,
                       tau_c=1.0, cos_tau_v=0.0, delta=3, lam=2.0, sigma=1.0, eps=0.05, rope_pairs=rope_pairs)
    st = ChunkStream.__new__(ChunkStream)  # layout only: no device buffers
    st.cfg = cfg
    return st


def _simulate(st, n_steps):
    """Contents of the sink and ring slots after each step, from the step's writes."""
    c = st.cfg
    ring = {}
    sink = None
    for n in range(n_steps):
        if n == 0:
            sink = 0
        else:
            ring[st.window_offset(n % c.window)] = n
        yield n, sink, dict(ring)


@pytest.mark.parametrize("k,window", [(1, 2), (2, 2), (3, 3), (2, 4)])
def test_live_window_segments_hold_exactly_the_last_chunks(k, window):
    st = _stream(k=k, window=window)
    c = st.cfg
    for n, sink, ring in _simulate(st, 40):
        segs = st.segments(n)
        assert segs[0] == (0, c.Nc, api.SEG_SINK, 0) and sink == 0
        live = {off for off, length, kind, _ in segs if kind == api.SEG_WINDOW and length > 0}
        assert live == set(ring)
        # the live ring slots hold the newest min(n, W) chunks, the sink excluded
        assert sorted(ring[o] for o in live) == list(range(max(1, n - window + 1), n + 1))
        # every ring slot is a full chunk or empty, and slots never overlap
        spans = sorted((off, off + length) for off, length, _, _ in segs if length > 0)
        assert all(b0 <= a1 for (_, b0), (a1, _) in zip(spans, spans[1:]))
        assert spans[-1][1] <= c.n_keys
        assert [s for s in segs if s[2] == api.SEG_RETRIEVED] == [
            ((1 + r) * c.Nc, c.Nc, api.SEG_RETRIEVED, r) for r in range(k)]


@pytest.mark.parametrize("window", [1, 2, 3])
def test_window_extension_is_the_newest_chunk_outside_window_and_sink(window):
    st = _stream(window=window)
    for n, _, ring in _simulate(st, 30):
        cached = set(ring.values()) | {0}
        older = [m for m in range(n + 1) if m not in cached]
        assert st.ext_first(n) == (max(older) if older else -1)


@pytest.mark.parametrize("k,window", [(1, 2), (2, 2), (3, 4)])
def test_repacked_slots_sit_just_before_the_window(k, window):
    """Slot r's frame f moves to pos_slot0 + r pos_stride + f; with the window's
    chunks at their own positions m F + f, the retrieved and window frames form one
    run of consecutive positions ending at the current chunk's last frame."""
    st = _stream(k=k, window=window, rope_pairs=4)
    c = st.cfg
    for n, _, ring in _simulate(st, 25):
        if n < window:
            continue  # the window is not full yet
        rp = st.rope(n)
        assert rp.pos_stride == c.F and rp.frame_pos0 == 0 and rp.pairs == 4
        slot_pos = [rp.pos_slot0 + r * rp.pos_stride + f for r in range(k) for f in range(c.F)]
        window_pos = sorted(m * c.F + f for m in ring.values() for f in range(c.F))
        run = slot_pos + window_pos
        assert run == list(range(run[0], run[0] + len(run)))
        assert run[-1] == (n + 1) * c.F - 1
    assert _stream(rope_pairs=0).rope(10) is None
