"""apc_upload (host-to-device copy executed by the SMs) and
apc_set_reserved_sms on the GPU: bytes land exactly, for every alignment
case, source kind and CTA count, and the step's results do not depend on
the SMs left free."""
import ctypes

import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

import paper_2609_18178_gb300 as apc  # noqa: E402


def pinned_bytes(n, seed):
    rng = np.random.default_rng(seed)
    h = torch.empty(n, dtype=torch.uint8, pin_memory=True)
    h.copy_(torch.from_numpy(rng.integers(0, 256, size=n, dtype=np.uint8)))
    return h


@pytest.mark.parametrize("ctas", [0, 1, 7])
def test_segments_of_every_alignment_land_exactly(ctas):
    """Mutually aligned segments with heads and tails, mutually misaligned
    ones, tiny and multi-tile ones, between guard bands that stay untouched."""
    h = pinned_bytes(3 << 20, 1)
    d = torch.full((3 << 20,), 0xA5, dtype=torch.uint8, device="cuda")
    cases = [(0, 0, 1 << 20), (5, 5, 700_001), (3, 11, 9_999), (16, 32, 15), (7, 7, 1), (1, 2, 3), (64, 64, 0),
             (13, 13, 131_073)]
    segs, spans, at = [], [], 64
    for so, do, n in cases:
        src = h[so + at:]
        dst = d[do + at:]
        segs.append(apc.Segment(dst, src, n))
        spans.append((do + at, so + at, n))
        at += max(n, 1) + 4096
    apc.upload(segs, ctas)
    torch.cuda.synchronize()
    got, want = d.cpu().numpy(), h.numpy()
    mask = np.zeros(got.size, dtype=bool)
    for do, so, n in spans:
        assert np.array_equal(got[do:do + n], want[so:so + n]), (do, so, n)
        mask[do:do + n] = True
    assert np.all(got[~mask] == 0xA5)                           # nothing outside the destinations


def test_more_segments_than_one_launch():
    h = pinned_bytes(1 << 20, 2)
    d = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    segs = [apc.Segment(d[i * 1000:], h[i * 1000 + 3:], 997) for i in range(1000)]
    apc.upload(apc.prepare_segments(segs), 3)
    torch.cuda.synchronize()
    got, want = d.cpu().numpy(), h.numpy()
    for i in range(1000):
        assert np.array_equal(got[i * 1000:i * 1000 + 997], want[i * 1000 + 3:i * 1000 + 1000])


def test_device_and_pageable_sources():
    d = torch.zeros(1 << 16, dtype=torch.uint8, device="cuda")
    s = torch.arange(1 << 16, dtype=torch.int32, device="cuda").to(torch.uint8)
    apc.upload([apc.Segment(d, s)], 2)
    torch.cuda.synchronize()
    assert torch.equal(d, s)
    pageable = np.random.default_rng(3).integers(0, 256, size=1 << 16, dtype=np.uint8)
    dev = torch.cuda.current_device()
    value = ctypes.c_int(0)
    cudart = ctypes.CDLL("libcudart.so")
    assert cudart.cudaDeviceGetAttribute(ctypes.byref(value), 88, dev) == 0  # cudaDevAttrPageableMemoryAccess
    seg = [apc.Segment(d, pageable.ctypes.data, pageable.size)]
    if value.value:
        apc.upload(seg, 2)
        torch.cuda.synchronize()
        assert np.array_equal(d.cpu().numpy(), pageable)
    else:
        with pytest.raises(apc.ApcError) as e:
            apc.upload(seg, 2)
        assert e.value.status == 1


def test_rejected_destinations():
    h = pinned_bytes(4096, 4)
    d = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    with pytest.raises(apc.ApcError) as e:                     # a host destination
        apc.upload([apc.Segment(h.data_ptr(), d.data_ptr(), 64)])
    assert e.value.status == 1
    with pytest.raises(apc.ApcError) as e:                     # overlapping destinations
        apc.upload([apc.Segment(d[0:], h, 100), apc.Segment(d[64:], h, 100)])
    assert e.value.status == 1
    with pytest.raises(apc.ApcError) as e:                     # a source overlapping a destination
        apc.upload([apc.Segment(d[0:], d[1000:], 100), apc.Segment(d[1050:], h, 100)])
    assert e.value.status == 1


@pytest.mark.parametrize("reserved", [16, 151, 1024])
def test_reserved_sms_do_not_change_results(reserved):
    from test_gpu_parity import assert_same, gen, run_small
    try:
        apc.set_reserved_sms(reserved)
        tensors = [gen(n, off, 2) for n, off in ((300_007, (1 << 32) - 9), (77, 400_000))]
        devs, dgot, ref, dref = run_small(tensors, 2)
        assert_same(devs, dgot, ref, dref)
        bufs = [b for dd, t in zip(devs, tensors)
                for b in apc.state_buffers(dd["p"], dd["m"], dd["v"], dd["w"], t["goff"])]
        assert apc.digests_to_host(apc.digest(bufs, 4)) == dref
    finally:
        apc.set_reserved_sms(0)


def test_upload_commit_digest_captured_in_one_graph():
    """Upload of the gradient from pinned host memory, the step and the
    verification digest, captured once as a CUDA graph; each replay uploads
    the gradient the host wrote since, and the chained state equals the
    oracle's."""
    import synth
    from test_gpu_parity import assert_same, dev, gen
    specs = [(40_000, (1 << 32) - 20_000), (3, 300_000), (9_999, 300_003)]
    tensors = [gen(n, off, 1) for n, off in specs]
    devs, entries, hosts, segs = [], [], [], []
    for t in tensors:
        d = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=torch.zeros(t["p"].size, dtype=torch.int16,
                                                                            device="cuda"),
                 w=torch.zeros(t["p"].size, dtype=torch.int16, device="cuda"))
        devs.append(d)
        entries.append(apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], t["goff"]))
        h = torch.zeros(t["p"].size, dtype=torch.int16, pin_memory=True)
        hosts.append(h)
        segs.append(apc.Segment(d["g"], h))
    vb = [b for e in entries for b in apc.state_buffers(e.p, e.m, e.v, e.w, e.global_offset)]
    out_c = torch.empty(4, dtype=torch.int64, device="cuda")
    out_v = torch.empty(4, dtype=torch.int64, device="cuda")
    tab, vtab, seg = apc.prepare_table(entries), apc.prepare_buffers(vb), apc.prepare_segments(segs)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):                       # first calls outside capture (per-device queries)
        apc.upload(seg, 4, stream=s)
        apc.commit_step(tab, 7, stream=s, out=out_c)
    torch.cuda.synchronize()
    for t, d in zip(tensors, devs):                  # back to the generated state
        for k in "pmv":
            d[k].copy_(torch.from_numpy(t[k]).cuda())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            apc.upload(seg, 4, stream=s)
            apc.commit_step(tab, 7, stream=s, out=out_c)
            apc.digest(vtab, 4, stream=s, out=out_v)
    torch.cuda.synchronize()
    for t, d in zip(tensors, devs):
        for k in "pmv":
            d[k].copy_(torch.from_numpy(t[k]).cuda())
    h8 = oracle.resolve_hparams(oracle.DEFAULT_HP, 7)
    ref = [dict(p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy(), goff=t["goff"]) for t in tensors]
    for rep in range(3):                             # a new gradient from the host before every replay
        for (n, off), h, r in zip(specs, hosts, ref):
            g = synth.grad(n, off, 10 + rep)
            h.copy_(torch.from_numpy(g.view(np.int16)))
            r["g"] = g
        graph.replay()
        torch.cuda.synchronize()
        ws, dref = oracle.commit_table(ref, h8)
        for r, wv in zip(ref, ws):
            r["w"] = wv
        assert_same(devs, apc.digests_to_host(out_c), ref, dref)
        assert apc.digests_to_host(out_v) == dref
        for d, r in zip(devs, ref):
            assert np.array_equal(d["g"].cpu().numpy().view(np.uint16), r["g"])
