"""Replica verification on the GPU: replica processes
of one hybrid-sharding replication group commit identical shards, verify,
and agree over the Gloo control plane; a bit flipped in one replica's HBM
state through a host-side copy is then seen by every replica."""
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)


def test_two_replicas_agree_then_catch_a_flipped_bit():
    import bench
    r = bench.replica_check(2, "c3", flip=1, timeout_s=300)
    assert "error" not in r, r
    assert r["commit_digests_equal"] and r["clean_agreed"]
    assert r["flip_detected_by_all"]
    assert tuple(r["flip_diagnosis"]) == ("state digests of shard 0", [0, 1])
