"""Row sharding of the corpus and the exchange step of a sharded search, on
the CPU: shard ranges, and two gloo ranks that each search their own rows with
the oracle, all-gather their top-k and merge, against the oracle's search of
the whole corpus ("sharded merge == global")."""
import os
import socket

import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from paper_2607_16973_gb300.shard import shard_rows
from parity import merge_candidates


@pytest.mark.parametrize("n", [0, 1, 63, 64, 65, 1000, 999_000])
@pytest.mark.parametrize("world", [1, 2, 3, 8])
@pytest.mark.parametrize("align", [1, 32, 64])
def test_shard_rows_partition(n, world, align):
    """Contiguous, disjoint, covering [0, n), aligned starts, balanced to one block."""
    r = [shard_rows(n, world, i, align) for i in range(world)]
    assert r[0][0] == 0 and r[-1][1] == n
    for (a, b), (c, _) in zip(r, r[1:]):
        assert b == c
    for a, b in r:
        assert a <= b and a % align == 0
    sizes = [b - a for a, b in r]
    assert max(sizes) - min(sizes) <= align


def test_sharded_search_refuses_an_id_map():
    from paper_2607_16973_gb300 import shard
    with pytest.raises(ValueError, match="no id map"):
        shard.sharded_search(None, None, None, 4, None, None, 5, 0, idmap=object())


def test_shard_rows_rejects_bad_rank():
    with pytest.raises(ValueError):
        shard_rows(10, 2, 2)
    with pytest.raises(ValueError):
        shard_rows(10, 0, 0)


def _problem(filtered):
    n, d, bits, nq, k = 1000, 64, 4, 4, 10
    X = synth.gaussian_rows(n, d, seed=11)
    R = O.rotation(d, 5).astype(np.float32)
    cb = O.codebook(d, bits)
    enc = O.encode(X, R, cb.centroids32, cb.boundaries32, bits)
    Q = synth.gaussian_rows(nq, d, seed=12)
    ten = None
    off = ids = None
    if filtered:
        # tenant 7 holds only 3 rows, all in the second shard: the first
        # shard returns nothing for query 0 and pads with -1
        ten = np.full(n, 1, np.uint32)
        ten[::2] = 2
        ten[[700, 701, 999]] = 7
        off = np.array([0, 1, 3, 4, 6], np.int64)
        ids = np.array([7, 1, 7, 2, 1, 2], np.uint32)
    return dict(n=n, d=d, bits=bits, k=k, Q=Q, R=R, c=cb.centroids32, enc=enc, ten=ten, off=off, ids=ids)


def _rank_main(rank, world, port, filtered, out_dir):
    import torch
    import torch.distributed as dist
    from paper_2607_16973_gb300.shard import gather_topk
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        P = _problem(filtered)
        lo, hi = shard_rows(P["n"], world, rank, 64)
        ten = P["ten"][lo:hi] if filtered else None
        res = O.search(P["Q"], P["R"], P["c"], P["bits"], P["enc"].packed[lo:hi], P["enc"].scale[lo:hi], P["k"],
                       P["d"], ten, P["off"], P["ids"])
        ci, cs = gather_topk(torch.from_numpy(res.ids), torch.from_numpy(res.scores), lo)
        np.save(os.path.join(out_dir, f"ids{rank}.npy"), ci.numpy())
        np.save(os.path.join(out_dir, f"sc{rank}.npy"), cs.numpy())
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("filtered", [False, True])
def test_gloo_two_ranks_sharded_merge_equals_global(tmp_path, filtered):
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), filtered, str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    P = _problem(filtered)
    ref = O.search(P["Q"], P["R"], P["c"], P["bits"], P["enc"].packed, P["enc"].scale, P["k"], P["d"],
                   P["ten"], P["off"], P["ids"])
    gathered = [(np.load(tmp_path / f"ids{r}.npy"), np.load(tmp_path / f"sc{r}.npy")) for r in range(world)]
    for ci, cs in gathered[1:]:  # every rank holds the same gathered lists
        np.testing.assert_array_equal(ci, gathered[0][0])
        np.testing.assert_array_equal(cs, gathered[0][1])
    ids, sc = merge_candidates(gathered[0][0], gathered[0][1], P["k"])
    np.testing.assert_array_equal(ids, ref.ids)
    np.testing.assert_array_equal(sc, ref.scores)
    if filtered:  # query 0 allows only tenant 7: three rows, then padding
        assert sorted(ids[0, :3]) == [700, 701, 999]
        assert np.all(ids[0, 3:] == -1)


def _rank_lost_main(rank, world, port, out_dir):
    """Rank 1 dies before the exchange; rank 0 must learn of it from the
    collective (process-group timeout or closed connection), not hang."""
    import datetime
    import torch
    import torch.distributed as dist
    from paper_2607_16973_gb300.shard import gather_topk
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=10))
    if rank == 1:
        os._exit(3)  # the shard is lost between steps, with nothing in flight
    ids = torch.zeros((2, 5), dtype=torch.int64)
    scores = torch.zeros((2, 5), dtype=torch.float32)
    try:
        gather_topk(ids, scores, 0)
        outcome = "completed"
    except Exception as e:  # noqa: BLE001 - any collective error is the detection
        outcome = "detected: " + type(e).__name__
    with open(os.path.join(out_dir, "rank0.txt"), "w") as f:
        f.write(outcome)
    os._exit(0)


def test_gloo_lost_rank_is_detected(tmp_path):
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    port = _free_port()
    procs = [ctx.Process(target=_rank_lost_main, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=60)
    alive = [p for p in procs if p.is_alive()]
    for p in alive:
        p.kill()
    assert not alive, "a rank hung after its peer was lost"
    assert procs[1].exitcode == 3
    assert (tmp_path / "rank0.txt").read_text().startswith("detected")
