"""Multi-rank host logic on CPU (gloo, world size 2): the by-sequence split of a
ragged batch (paper_2608_08794_gb300.shard) with real work on each rank, the
max-over-ranks timing and whole-job value of bench.py, and the reference arm
under torchrun (rank 0 prints the only line, rank 1 exits 0).

The split is checked with the oracle standing in for each rank's GPU: every
rank scores, selects and compacts only its own sequences, maps its kept
indices back to the whole batch, and the merged result must equal the oracle
run over the whole batch at once (Sec. 3.2 scores and selects per sequence, so
the split may change nothing)."""

import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = 10.0 + 5.0 * rank                      # rank 1 is the slow one
    got = bench.max_over_ranks(ms, dist, "cpu")
    dist.barrier()
    out[rank] = got
    dist.destroy_process_group()


def test_max_over_ranks_with_two_gloo_ranks():
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    assert dict(out) == {0: 15.0, 1: 15.0}


def test_whole_job_value_counts_every_replica():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.whole_job_value(231000, 1, 2.5) == pytest.approx(231000 / 2.5e-3)
    assert bench.whole_job_value(231000, 4, 2.5) == pytest.approx(4 * 231000 / 2.5e-3)
    assert bench.max_over_ranks(3.0, None, "cpu") == 3.0


def test_reference_arm_under_torchrun_prints_one_line_from_rank_zero():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    r = subprocess.run(cmd, capture_output=True, text=True, cwd=ROOT, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [json.loads(x) for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    line = lines[0]
    assert line["impl"] == "reference" and line["value"] > 0 and line["cpu_baseline"]["cores"] == 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["n_gpus"] == 2


def _ragged_batch(seed=3, n=7, hq=4, hkv=2):
    """A small ragged batch: 7 sequences of 30..400 tokens, audio/visual/other mixed,
    1..9 query rows each, bf16 keys and queries, a third plane of wider rows."""
    sys.path.insert(0, ROOT)
    from synth.gen import f32_to_bf16_bits
    rng = np.random.default_rng(seed)
    lens = rng.integers(30, 400, n)
    nqs = rng.integers(1, 10, n)
    mod = rng.choice([0, 1, 2], int(lens.sum()), p=[0.05, 0.25, 0.7]).astype(np.uint8)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    cuq = np.concatenate([[0], np.cumsum(nqs)]).astype(np.int32)
    k = f32_to_bf16_bits(rng.standard_normal((int(cu[-1]), hkv, 128)).astype(np.float32))
    q = f32_to_bf16_bits(rng.standard_normal((int(cuq[-1]), hq, 128)).astype(np.float32))
    hidden = rng.integers(0, 1 << 16, (int(cu[-1]), 40)).astype(np.uint16)
    na = np.array([(mod[cu[b]:cu[b + 1]] == 1).sum() for b in range(n)], np.int32)
    nv = np.array([(mod[cu[b]:cu[b + 1]] == 2).sum() for b in range(n)], np.int32)
    ratios = rng.integers(200, 601, (n, 2)) / 1000.0
    return dict(mod=mod, cu=cu, cuq=cuq, k=k, q=q, hidden=hidden, na=na, nv=nv, ratios=ratios, hq=hq, hkv=hkv)


def _shard_rank(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import oracle
    from paper_2608_08794_gb300.shard import plan_by_sequence, SequenceShard
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    d = _ragged_batch()
    counts = oracle.step_keep_counts([tuple(r) for r in d["ratios"]], list(zip(d["na"], d["nv"])))
    plan = plan_by_sequence(d["cu"], world)
    sh = SequenceShard(plan[rank], d["cu"], d["cuq"], d["na"], d["nv"])
    # this rank's step, on its own sequences only (the oracle standing in for its GPU)
    res = oracle.prune_step(sh.query_rows(d["q"]), sh.tokens(d["k"]), sh.cu_seqlens, sh.cu_qlens,
                            sh.tokens(d["mod"]), d["hq"], d["hkv"], [tuple(c) for c in sh.keep_counts(counts)],
                            planes=[sh.tokens(d["k"]), sh.tokens(d["hidden"])])
    mine = {"seq_ids": sh.seq_ids.tolist(), "keep": sh.to_global(res["keep_idx"]).tolist(),
            "new_cu": res["cu_seqlens"].tolist(), "scores": res["scores"].tolist(),
            "token_index": sh.token_index.tolist(), "k_rows": res["planes"][0].tolist(),
            "h_rows": res["planes"][1].tolist()}
    got = [None] * world
    dist.all_gather_object(got, mine)          # verification only: the step itself exchanges nothing
    if rank == 0:
        out["parts"] = got
    dist.barrier()
    dist.destroy_process_group()


def test_sequence_split_over_two_gloo_ranks_equals_the_whole_batch():
    sys.path.insert(0, ROOT)
    import oracle
    from paper_2608_08794_gb300.shard import SequenceShard, merge_keep, merge_cu_seqlens
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_shard_rank, args=(world, port, out), nprocs=world, join=True)
    parts = out["parts"]
    d = _ragged_batch()
    B = len(d["cu"]) - 1
    # every sequence on exactly one rank, both ranks busy
    ids = sorted(i for p in parts for i in p["seq_ids"])
    assert ids == list(range(B)) and all(p["seq_ids"] for p in parts)
    counts = oracle.step_keep_counts([tuple(r) for r in d["ratios"]], list(zip(d["na"], d["nv"])))
    whole = oracle.prune_step(d["q"], d["k"], d["cu"], d["cuq"], d["mod"], d["hq"], d["hkv"],
                              [tuple(c) for c in counts], planes=[d["k"], d["hidden"]])
    # kept indices and offsets
    keep = merge_keep([p["keep"] for p in parts])
    np.testing.assert_array_equal(keep, whole["keep_idx"])
    shards = [SequenceShard(p["seq_ids"], d["cu"], d["cuq"], d["na"], d["nv"]) for p in parts]
    np.testing.assert_array_equal(merge_cu_seqlens(shards, [p["new_cu"] for p in parts], B), whole["cu_seqlens"])
    # scores: each rank's scores land on the whole batch's tokens unchanged
    scores = np.zeros(int(d["cu"][-1]))
    for p in parts:
        scores[np.asarray(p["token_index"])] = p["scores"]
    np.testing.assert_array_equal(scores, whole["scores"])
    # compacted rows: each rank's rows are the whole batch's rows of its kept tokens
    for p in parts:
        pos = np.searchsorted(whole["keep_idx"], np.asarray(p["keep"]))
        np.testing.assert_array_equal(np.asarray(p["k_rows"], np.uint16), whole["planes"][0][pos])
        np.testing.assert_array_equal(np.asarray(p["h_rows"], np.uint16), whole["planes"][1][pos])


def test_sequence_plan_balances_the_ragged_workload():
    sys.path.insert(0, ROOT)
    from paper_2608_08794_gb300.shard import plan_by_sequence
    from synth import workload
    wl = workload("7b_ragged16")
    cu = wl.cu_seqlens()
    lens = np.diff(cu)
    for world in (1, 2, 3, 4, 8, 16, 20):
        plan = plan_by_sequence(cu, world)
        assert len(plan) == world
        assert sorted(np.concatenate(plan).tolist()) == list(range(wl.num_seqs))
        assert all(np.all(np.diff(p) > 0) for p in plan)
        loads = [int(lens[p].sum()) for p in plan]
        # greedy longest-first: no rank exceeds the mean load by more than one sequence
        assert max(loads) <= lens.sum() / world + lens.max()
        if world <= wl.num_seqs:
            assert min(loads) > 0
        assert plan_by_sequence(cu, world)[0].tolist() == plan[0].tolist()     # deterministic
    two = plan_by_sequence(cu, 2)
    assert abs(int(lens[two[0]].sum()) - int(lens[two[1]].sum())) <= lens.max()


def test_shard_maps_tokens_and_rejects_bad_ids():
    sys.path.insert(0, ROOT)
    from paper_2608_08794_gb300.shard import SequenceShard, merge_keep
    cu, cuq = [0, 3, 3, 7, 12], [0, 1, 1, 3, 4]
    sh = SequenceShard([0, 2, 3], cu, cuq, [1, 0, 2, 2], [1, 0, 1, 2])
    assert sh.cu_seqlens.tolist() == [0, 3, 7, 12] and sh.cu_qlens.tolist() == [0, 1, 3, 4]
    assert sh.token_index.tolist() == [0, 1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11]
    sh = SequenceShard([1, 3], cu, cuq, [1, 0, 2, 2], [1, 0, 1, 2])
    assert sh.token_index.tolist() == [7, 8, 9, 10, 11] and sh.q_index.tolist() == [3]
    assert sh.to_global([0, 4]).tolist() == [7, 11]
    with pytest.raises(ValueError):
        SequenceShard([2, 1], cu, cuq, [1, 0, 2, 2], [1, 0, 1, 2])
    with pytest.raises(ValueError):
        merge_keep([[1, 2], [2, 5]])


def test_multicore_oracle_baseline_keeps_what_the_single_threaded_oracle_keeps():
    """bench.py's multi-core CPU baseline splits the oracle's scoring over KV head groups and
    query-row chunks and recombines the parts (the mean over heads and rows is linear): on a
    20-s prefix of the 10-minute schedule it keeps exactly the tokens the plain oracle keeps."""
    sys.path.insert(0, ROOT)
    import bench
    one = bench.run_oracle("7b_10min", 20, 1)
    many = bench.run_oracle_pool("7b_10min", 20, 3)
    assert (one["kept"], one["kept_sum"], one["mm"]) == (many["kept"], many["kept_sum"], many["mm"])
