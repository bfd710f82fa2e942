"""Pointer ownership at the C ABI on a GPU: buffers that are not memory of
the current device (page-locked or pageable host memory) are refused with
APC_EINVAL before anything is enqueued, so the caller's output is left as it
was."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # the CUDA path has no fallback: without a GPU these tests cannot run
    pytest.skip("no CUDA device", allow_module_level=True)

import paper_2609_18178_gb300 as apc  # noqa: E402

N = 4096
SENTINEL = 0x5A5A5A5A


def _device_set():
    d = {k: torch.zeros(N, dtype=torch.float32, device="cuda") for k in "pmv"}
    d["g"] = torch.zeros(N, dtype=torch.int16, device="cuda")
    d["w"] = torch.zeros(N, dtype=torch.int16, device="cuda")
    return d


def _refused(call):
    with pytest.raises(apc.ApcError) as ei:
        call()
    assert ei.value.status == 1, ei.value
    return str(ei.value)


def test_host_pointers_are_refused_before_launch():
    d = _device_set()
    out = torch.full((8,), SENTINEL, dtype=torch.int64, device="cuda")
    pinned = torch.zeros(N, dtype=torch.float32).pin_memory()
    pageable = np.zeros(N, dtype=np.float32)
    for bad in (pinned.data_ptr(), pageable.ctypes.data):
        for field in "pmvgw":
            e = dict(d)
            e[field] = bad
            msg = _refused(lambda: apc.commit_step([apc.TensorEntry(e["p"], e["m"], e["v"], e["g"], e["w"], 0,
                                                                    n=N)], 1, out=out[:4]))
            assert "table[0].%s" % field in msg
        _refused(lambda: apc.digest([apc.BufferEntry(bad, 0, 0, apc.F32, n=N)], 1, out=out[4:5]))
        _refused(lambda: apc.count_nonzero([apc.BufferEntry(bad, 0, 0, apc.F32, n=N)], 1, out=out[5:6]))
    host_out = torch.zeros(4, dtype=torch.int64).pin_memory()
    msg = _refused(lambda: apc.commit_step([apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 0)], 1,
                                           out=host_out.data_ptr()))
    assert "out_digests" in msg
    _refused(lambda: apc.digest(apc.state_buffers(d["p"], d["m"], d["v"], d["w"]), 4, out=host_out.data_ptr()))
    torch.cuda.synchronize()
    assert out.cpu().tolist() == [SENTINEL] * 8      # nothing was zeroed or launched
    assert int(host_out.abs().sum()) == 0


def test_device_pointers_still_pass():
    d = _device_set()
    out = apc.commit_step([apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 0)], 1)
    ver = apc.digest(apc.state_buffers(d["p"], d["m"], d["v"], d["w"]), 4)
    assert apc.digests_to_host(out) == apc.digests_to_host(ver)


def test_output_overlapping_a_buffer_is_refused():
    d = _device_set()
    _refused(lambda: apc.commit_step([apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 0)], 1,
                                     out=d["m"][8:16].view(torch.int64)))
    _refused(lambda: apc.digest(apc.state_buffers(d["p"], d["m"], d["v"], d["w"]), 4,
                                out=d["v"][:8].view(torch.int64)))
