"""The long-horizon loop-closure stream (200 chunk steps on a closed camera loop,
Wan-1.3B head shape, 30 layers, k = 2) through ChunkStream: every step's
retrieval must match the oracle bit-exactly and its correspondences within the
boundary band; the cache invariants (sink = chunk 0, window = newest chunks,
retrieved slots = the retrieved chunks' own K/V) must hold; attention is compared
with the oracle on sampled steps, layers and query rows.  The bank keeps the K/V of
all 200 chunks (200 slabs, 172 GB at 30 layers); a second stream with a pool of 16
slabs checks that a chunk whose slab was reused is never retrieved."""

import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2607_21848_gb300 import stream as crs
from tests import _gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_21848_gb300 import build
    build.build()


def test_loop_stream_200_steps():
    wl = synth.make_workload(5)
    cfg = crs.StreamConfig(L=wl.L, H=wl.H, d=wl.d, F=wl.F, h=wl.h, w=wl.w, k=wl.k, window=2,
                           capacity=wl.bank_size, num_slabs=wl.bank_size, E=wl.E, w_v=wl.w_v, tau_c=wl.tau_c,
                           cos_tau_v=wl.cos_tau_v, delta=wl.delta, lam=wl.lam, sigma=wl.sigma, eps=wl.eps)
    st = crs.ChunkStream(cfg)
    Nc = cfg.Nc
    g = torch.Generator(device="cuda").manual_seed(5)
    s = wl.qkv_scale
    nbuf = 3
    kv_new = [((torch.randn(cfg.L, Nc, cfg.H, cfg.d, generator=g, device="cuda") * s).bfloat16(),
               (torch.randn(cfg.L, Nc, cfg.H, cfg.d, generator=g, device="cuda") * s).bfloat16()) for _ in range(nbuf)]
    q = (torch.randn(cfg.L, Nc, cfg.H, cfg.d, generator=g, device="cuda") * s).bfloat16()
    o = torch.empty_like(q)
    lse = torch.empty(cfg.L, cfg.H, Nc, device="cuda")
    check_attn = {1, 2, 3, 150, 151, 199}
    layers, heads = [0, 29], [0, 7]
    host_kv = [(kb[layers][:, :, heads].double().cpu().numpy(), vb[layers][:, :, heads].double().cpu().numpy())
               for kb, vb in kv_new]
    host_q = q[layers][:, :, heads].double().cpu().numpy()
    n_closed = 0
    for n in range(wl.bank_size):
        fr = wl.bank_frames[n]
        dep = torch.from_numpy(wl.depth_of(n)).cuda()
        kn, vn = kv_new[n % nbuf]
        st.step(n, synth.frame_records(fr), dep, kn, vn, q, o, lse)
        torch.cuda.synchronize()
        assert st.status.item() == 0
        # retrieval: bit-exact indices and count
        ext = st.ext_first(n)
        oi, os_, oc, slots = _gpu.oracle_retrieve(wl, bank_count=n + 1, n=n, ext_first=ext, ext_min=1)
        gi = st.idx.cpu().numpy()
        assert int(st.count.item()) == oc, n
        np.testing.assert_array_equal(gi, slots)
        np.testing.assert_array_equal(st.score.cpu().numpy()[:oc], os_[:oc])
        n_closed += oc > 0
        # cache invariants, against the chunks' K/V buffers
        assert torch.equal(st.cache.k[:, :Nc], kv_new[0][0])  # sink = chunk 0
        for m in range(max(1, n - 1), n + 1):
            off = st.window_offset(m % 2)
            assert torch.equal(st.cache.k[:, off:off + Nc], kv_new[m % nbuf][0])
            assert torch.equal(st.cache.v[:, off:off + Nc], kv_new[m % nbuf][1])
        for r, j in enumerate(slots):
            if j >= 0:  # the retrieved chunk's own K/V (chunk j was written from buffer j % nbuf)
                off = st.slot_offset(r)
                src = kv_new[j % nbuf]
                assert torch.equal(st.cache.k[:, off:off + Nc], src[0])
                assert torch.equal(st.cache.v[:, off:off + Nc], src[1])
        # correspondences
        ocor = _gpu.oracle_correspond(wl, slots, oc, cur=fr, depth_cur=wl.depth_of(n))
        r = _gpu.compare_correspondence(wl, ocor, st.uv.cpu().numpy().astype(np.float64), st.cell.cpu().numpy(),
                                        st.valid.cpu().numpy(), wl.eps, depth_cur=wl.depth_of(n))
        assert r["bad_valid"] == 0 and r["bad_cell"] == 0 and r["uv_err"] <= 1e-3, (n, r)
        if n in check_attn:
            # oracle inputs come from the seeded inputs only: its own retrieval and
            # correspondences, and a cache assembled from the chunks' K/V buffers
            uv, _, valid, _, _, _ = ocor
            agree = (st.valid.cpu().numpy().astype(bool) == valid).all(axis=1)
            rows = np.random.default_rng(n).choice(np.nonzero(agree)[0], 128, replace=False)
            rows.sort()
            Kx = np.zeros((len(layers), cfg.n_keys, len(heads), cfg.d))
            Vx = np.zeros_like(Kx)
            Kx[:, :Nc], Vx[:, :Nc] = host_kv[0]
            for rr, j in enumerate(slots):
                if j >= 0:
                    off = st.slot_offset(rr)
                    Kx[:, off:off + Nc], Vx[:, off:off + Nc] = host_kv[j % nbuf]
            for m in range(max(1, n - 1), n + 1):
                off = st.window_offset(m % 2)
                Kx[:, off:off + Nc], Vx[:, off:off + Nc] = host_kv[m % nbuf]
            uvo = uv.copy()
            uvo[~valid] = 0.0
            Oo, lo = oracle.attention(host_q, Kx, Vx, uvo.astype(np.float32).astype(np.float64), valid,
                                      st.segments(n), cfg.h, cfg.w, cfg.F, cfg.lam, cfg.sigma, slot_chunks=slots,
                                      rows=rows)
            Og = o[layers][:, :, heads].float().cpu().numpy()[:, rows]
            err, rel, rms = _gpu.attn_errors(Og, Oo)
            assert err <= 2e-2 and rel <= 2e-2, (n, err, rel)
            lg = lse[layers][:, heads].cpu().numpy()[:, :, rows]
            assert np.abs(lg - lo).max() <= 1e-3
    assert n_closed >= 40  # the loop closes after one lap and stays closed
    del st
    torch.cuda.empty_cache()


def test_loop_stream_with_a_small_slab_pool_never_gathers_a_reused_slab():
    """The same 200-step loop with 16 K/V slabs for 200 chunks (2 layers, 2 heads): chunk j's
    slab is reused by chunk j + 16, so from then on j is not retrievable.  Every step's
    retrieval equals the oracle's over the chunks still held, and every gathered slot holds
    its chunk's own K/V."""
    wl = synth.make_workload(5)
    P = 16
    cfg = crs.StreamConfig(L=2, H=2, d=wl.d, F=wl.F, h=wl.h, w=wl.w, k=wl.k, window=2, capacity=wl.bank_size,
                           num_slabs=P, E=wl.E, w_v=wl.w_v, tau_c=wl.tau_c, cos_tau_v=wl.cos_tau_v,
                           delta=wl.delta, lam=wl.lam, sigma=wl.sigma, eps=wl.eps)
    st = crs.ChunkStream(cfg)
    Nc = cfg.Nc
    g = torch.Generator(device="cuda").manual_seed(12)
    kv = [((torch.randn(2, Nc, 2, cfg.d, generator=g, device="cuda") * wl.qkv_scale).bfloat16(),
           (torch.randn(2, Nc, 2, cfg.d, generator=g, device="cuda") * wl.qkv_scale).bfloat16()) for _ in range(5)]
    q = kv[0][0].clone()
    o = torch.empty_like(q)
    closed_full = closed_held = 0
    for n in range(wl.bank_size):
        kn, vn = kv[n % 5]
        st.step(n, synth.frame_records(wl.bank_frames[n]), torch.from_numpy(wl.depth_of(n)).cuda(), kn, vn, q, o)
        torch.cuda.synchronize()
        assert st.status.item() == 0
        held = np.zeros(wl.bank_size, bool)
        held[max(0, n - P + 1):n + 1] = True
        _, _, oc, slots = _gpu.oracle_retrieve(wl, bank_count=n + 1, n=n, ext_first=st.ext_first(n), ext_min=1,
                                               resident=held)
        gi = st.idx.cpu().numpy()
        assert int(st.count.item()) == oc, n
        np.testing.assert_array_equal(gi, slots)
        for r, j in enumerate(gi):
            if j >= 0:
                assert held[j]
                off = st.slot_offset(r)
                assert torch.equal(st.cache.k[:, off:off + Nc], kv[j % 5][0])
                assert torch.equal(st.cache.v[:, off:off + Nc], kv[j % 5][1])
        closed_held += oc > 0
        closed_full += _gpu.oracle_retrieve(wl, bank_count=n + 1, n=n)[2] > 0
    # the loop's start (chunks 0-2) is long gone from the 16-slab pool when the camera returns
    assert closed_full >= 40 and closed_held < closed_full


def test_loop_stream_with_rope_repositioning_and_control_mirror():
    # the same 200-step loop with re-positioned retrieved keys and a control-branch cache
    # mirroring the retrieved slots (small head count; retrieval and gathers are what is checked)
    wl = synth.make_workload(5)
    cfg = crs.StreamConfig(L=2, H=2, d=wl.d, F=wl.F, h=wl.h, w=wl.w, k=wl.k, window=2, capacity=wl.bank_size,
                           num_slabs=wl.bank_size, E=wl.E, w_v=wl.w_v, tau_c=wl.tau_c, cos_tau_v=wl.cos_tau_v,
                           delta=wl.delta, lam=wl.lam, sigma=wl.sigma, eps=wl.eps, rope_pairs=22,
                           rope_interleaved=True, control_L=1)
    st = crs.ChunkStream(cfg)
    Nc = cfg.Nc
    g = torch.Generator(device="cuda").manual_seed(6)
    s = wl.qkv_scale
    nbuf = 3

    def rnd(L):
        return (torch.randn(L, Nc, cfg.H, cfg.d, generator=g, device="cuda") * s).bfloat16()

    kv = [(rnd(cfg.L), rnd(cfg.L)) for _ in range(nbuf)]
    ctl = [(rnd(1), rnd(1)) for _ in range(nbuf)]
    q = rnd(cfg.L)
    o = torch.empty_like(q)

    def rope_of(n):
        r = st.rope(n)
        return dict(channel0=r.channel0, pairs=r.pairs, theta=r.theta, interleaved=True, pos_slot0=r.pos_slot0,
                    pos_stride=r.pos_stride, frame_pos0=r.frame_pos0, F=cfg.F)

    checked = 0
    for n in range(wl.bank_size):
        fr = wl.bank_frames[n]
        dep = torch.from_numpy(wl.depth_of(n)).cuda()
        st.step(n, synth.frame_records(fr), dep, kv[n % nbuf][0], kv[n % nbuf][1], q, o,
                k_ctl=ctl[n % nbuf][0], v_ctl=ctl[n % nbuf][1])
        torch.cuda.synchronize()
        assert st.status.item() == 0
        _, _, oc, slots = _gpu.oracle_retrieve(wl, bank_count=n + 1, n=n, ext_first=st.ext_first(n), ext_min=1)
        np.testing.assert_array_equal(st.idx.cpu().numpy(), slots)
        # the window is never rotated: newest chunks byte-exact in both caches
        for m in range(max(1, n - 1), n + 1):
            off = st.window_offset(m % 2)
            assert torch.equal(st.cache.k[:, off:off + Nc], kv[m % nbuf][0])
            assert torch.equal(st.control_cache.k[:, off:off + Nc], ctl[m % nbuf][0])
        if not (n % 10 == 0 or 150 <= n <= 155):
            continue
        for r, j in enumerate(slots):
            if j < 0:
                continue
            owner = j % nbuf  # chunk j's own K/V
            off = st.slot_offset(r)
            for cache, src in ((st.cache, kv[owner]), (st.control_cache, ctl[owner])):
                host = np.stack([src[0].double().cpu().numpy(), src[1].double().cpu().numpy()])
                # slot r holds chunk j, read from a one-slab pool holding its K/V buffers
                ref = oracle.gather(host[None], np.array([-1] * r + [j]), 1, rope=rope_of(n))[r]
                got = cache.k[:, off:off + Nc]
                np.testing.assert_allclose(got.double().cpu().numpy(), ref[0], rtol=2.0 ** -8,
                                           atol=1e-6 * float(np.abs(host).max()))
                assert torch.equal(cache.v[:, off:off + Nc], src[1])
                checked += 1
    assert checked >= 40


def test_stream_resumes_from_a_checkpoint_bit_for_bit(tmp_path):
    # run 30 steps; checkpoint after step 19 to a file; a fresh stream restored from it
    # replays steps 20-29 with identical retrievals, correspondences and outputs
    wl = synth.make_workload(5)
    cfg = crs.StreamConfig(L=2, H=2, d=wl.d, F=wl.F, h=wl.h, w=wl.w, k=wl.k, window=2, capacity=30,
                           num_slabs=16, E=wl.E, w_v=wl.w_v, tau_c=1.0, cos_tau_v=-1.0, delta=wl.delta,
                           lam=wl.lam, sigma=wl.sigma, eps=wl.eps, rope_pairs=22, control_L=1)
    g = torch.Generator(device="cuda").manual_seed(8)

    def rnd(L):
        return (torch.randn(L, cfg.Nc, cfg.H, cfg.d, generator=g, device="cuda") * wl.qkv_scale).bfloat16()

    inputs = [(rnd(2), rnd(2), rnd(1), rnd(1)) for _ in range(30)]
    q = rnd(2)

    def run(st, steps):
        outs = []
        for n in steps:
            k, v, kc, vc = inputs[n]
            o = torch.empty_like(q)
            st.step(n, synth.frame_records(wl.bank_frames[n]), torch.from_numpy(wl.depth_of(n)).cuda(), k, v, q, o,
                    k_ctl=kc, v_ctl=vc)
            outs.append((st.idx.clone(), st.uv.clone(), st.valid.clone(), o))
        torch.cuda.synchronize()
        assert st.status.item() == 0
        return outs

    a = crs.ChunkStream(cfg)
    run(a, range(20))
    path = tmp_path / "stream.pt"
    torch.save({k: t.cpu() for k, t in a.state_dict().items()}, path)
    ref = run(a, range(20, 30))
    b = crs.ChunkStream(cfg)
    b.load_state_dict({k: t.cuda() for k, t in torch.load(path).items()})
    got = run(b, range(20, 30))
    assert any(int(r[0][0]) >= 0 for r in ref)  # the window-extension / retrieval slots are in use
    for (i0, u0, v0, o0), (i1, u1, v1, o1) in zip(ref, got):
        assert torch.equal(i0, i1) and torch.equal(v0, v1) and torch.equal(o0, o1)
        assert torch.equal(torch.nan_to_num(u0, nan=-9.0), torch.nan_to_num(u1, nan=-9.0))
    with pytest.raises(ValueError):
        b.load_state_dict({"cache.k": b.cache.k})


def test_graph_replayed_stream_matches_the_eager_stream_bit_for_bit():
    """The 200-step loop-closure stream (2 layers, 2 heads, k = 2, re-positioned keys, 200
    tracked K/V slabs, a bank of 600 so that the scoring runs on two blocks) through
    crc_chunk_step replayed from CUDA graphs, against the same stream through the separate
    entry points: every step's indices, count, scores, correspondences (raw bits, NaN
    included), cells, flags, output and LSE are identical.  A descriptor whose chunk lies
    outside the bank is then rejected on the device with CRC_STEP_BAD_DESCRIPTOR."""
    from paper_2607_21848_gb300 import _abi

    wl = synth.make_workload(5)
    cfg = crs.StreamConfig(L=2, H=2, d=wl.d, F=wl.F, h=wl.h, w=wl.w, k=wl.k, window=2, capacity=600, num_slabs=200,
                           E=wl.E, w_v=wl.w_v, tau_c=wl.tau_c, cos_tau_v=wl.cos_tau_v, delta=wl.delta, lam=wl.lam,
                           sigma=wl.sigma, eps=wl.eps, rope_pairs=22)
    eager, graph = crs.ChunkStream(cfg), crs.ChunkStream(cfg)
    assert graph.bank.workspace is not None  # 600 entries: the scoring's blocks meet in the workspace
    Nc = cfg.Nc
    g = torch.Generator(device="cuda").manual_seed(21)

    def rnd():
        return (torch.randn(cfg.L, Nc, cfg.H, cfg.d, generator=g, device="cuda") * wl.qkv_scale).bfloat16()

    kv = [(rnd(), rnd()) for _ in range(5)]
    q = rnd()
    o_e, o_g = torch.empty_like(q), torch.empty_like(q)
    lse_e = torch.empty(cfg.L, cfg.H, Nc, device="cuda")
    lse_g = torch.empty_like(lse_e)
    depth_buf = torch.empty(cfg.F, cfg.h, cfg.w, device="cuda")
    k_buf, v_buf = torch.empty_like(q), torch.empty_like(q)
    graph.capture(depth_buf, k_buf, v_buf, q, o_g, lse_g)
    bits = lambda t: t.view(torch.int32)  # noqa: E731
    closed = 0
    for n in range(wl.bank_size):
        fr = synth.frame_records(wl.bank_frames[n])
        dep = torch.from_numpy(wl.depth_of(n)).cuda()
        kn, vn = kv[n % 5]
        eager.step(n, fr, dep, kn, vn, q, o_e, lse_e)
        depth_buf.copy_(dep)
        k_buf.copy_(kn)
        v_buf.copy_(vn)
        graph.replay(n, fr)
        torch.cuda.synchronize()
        assert eager.status.item() == 0 and graph.status.item() == 0, n
        assert torch.equal(eager.idx, graph.idx) and torch.equal(eager.count, graph.count), n
        assert torch.equal(eager.score, graph.score), n
        assert torch.equal(bits(eager.uv), bits(graph.uv)), n
        assert torch.equal(eager.cell, graph.cell) and torch.equal(eager.valid, graph.valid), n
        assert torch.equal(o_e, o_g), n
        assert torch.equal(bits(lse_e), bits(lse_g)), n
        closed += int(graph.count.item()) > 0
    assert closed >= 40  # the loop closes after one lap: retrieved chunks go through the replayed step
    assert torch.equal(eager.bank.frames, graph.bank.frames) and torch.equal(eager.cache.k, graph.cache.k)
    # chunk 600 is outside a bank of 600: nothing is written, the status word says why
    frames_before = graph.bank.frames.clone()
    graph.replay(600, synth.frame_records(wl.bank_frames[0]))
    torch.cuda.synchronize()
    assert graph.status.item() == _abi.CRC_STEP_BAD_DESCRIPTOR
    assert int(graph.count.item()) == 0 and bool((graph.idx < 0).all())
    assert torch.equal(graph.bank.frames, frames_before)
