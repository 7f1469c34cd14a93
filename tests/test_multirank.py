"""The benchmark's multi-rank host logic on CPU: two gloo ranks.

The hot path shards by independent pipelines (weak scaling, no data-path
collective); the only cross-rank traffic is the barrier and the max/sum of
the timing and element counts."""
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    import seeded_inputs as SI
    r = bench.Ranks()
    r.init("gloo")
    try:
        r.barrier()
        mx = r.max(float(10 + rank))
        sm = r.sum(float(1 + rank))
        cfg = bench.rank_config(SI.SEVENTY_B, rank)
        q.put((rank, mx, sm, cfg["config_id"], cfg["n_canaries"]))
    finally:
        r.close()


def test_two_gloo_ranks():
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    q = mp.Queue()
    port = _free_port()
    procs = [mp.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[1] for o in out] == [11.0, 11.0]          # max over ranks
    assert [o[2] for o in out] == [3.0, 3.0]            # sum over ranks
    assert [o[3] for o in out] == [0, 1]                # distinct pipelines per rank
    assert out[0][4] == out[1][4] == 256                # same per-rank work (weak scaling)


def test_reference_arm_other_ranks_exit(capsys, monkeypatch):
    """Under torchrun only rank 0 runs the reference arm; others exit 0 silently."""
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    assert bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "1",
                       "--warmup", "0"]) == 0
    assert capsys.readouterr().out == ""
