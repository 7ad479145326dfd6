"""Multi-rank path on CPU: two gloo ranks each run the pruned block (oracle
arithmetic, CPU) on their own image shard; the gathered shards must equal the
unsharded batch, with no data-path collective needed."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import dora_synth as S
from paper_2609_34325_gb300.sharding import image_range, shard_packed


def test_image_ranges_cover_exactly_once():
    for batch in (0, 1, 7, 8, 256):
        for world in (1, 2, 3, 8):
            seen = []
            for r in range(world):
                lo, hi = image_range(batch, r, world)
                seen.extend(range(lo, hi))
                assert hi - lo in (batch // world, batch // world + 1)
            assert seen == list(range(batch))


def test_shard_packed_rebases_boundaries():
    cu = np.array([0, 5, 9, 20, 21])
    s0, s1 = shard_packed(cu, 0, 2), shard_packed(cu, 1, 2)
    assert s0["rows"] == (0, 9) and s0["cu_local"].tolist() == [0, 5, 9]
    assert s1["rows"] == (9, 21) and s1["cu_local"].tolist() == [0, 11, 12]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import oracle as O
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cfg = S.Config("tiny", batch=5, n_tokens=21, dim=128, heads=2, mlp_dim=256, depth=1,
                   prune_blocks=(0,), k_law="uniform", k_max=14)
    cu, ids = S.initial_layout(cfg)
    x = O.bf16_to_f64(S.activations_bf16(cfg, 3))
    wf = O.decode_weights(S.block_weights(cfg, 0, 3, random_affine=True))
    keeps, _ = S.keep_schedule(cfg, 3)
    scores = O.gather_scores(S.score_table(cfg, 0, 3), cu, ids)
    sh = shard_packed(cu, rank, world)
    r0, r1 = sh["rows"]
    lo, hi = sh["images"]
    res = O.pruned_block(x[r0:r1], sh["cu_local"], ids[r0:r1], wf, cfg.heads, cfg.ln_eps,
                         scores[r0:r1], keeps[0][lo:hi])
    mine = {"x": res["x_out"], "cu": res["cu_out"], "ids": res["ids_out"]}
    gathered = [None] * world
    dist.all_gather_object(gathered, mine)       # result collection only
    if rank == 0:
        full = O.pruned_block(x, cu, ids, wf, cfg.heads, cfg.ln_eps, scores, keeps[0])
        xs = np.concatenate([g["x"] for g in gathered])
        idss = np.concatenate([g["ids"] for g in gathered])
        counts = np.concatenate([np.diff(g["cu"]) for g in gathered])
        ok = (np.array_equal(xs, full["x_out"]) and np.array_equal(idss, full["ids_out"])
              and np.array_equal(counts, np.diff(full["cu_out"])))
        with open(os.path.join(out_dir, "ok"), "w") as f:
            f.write("1" if ok else "0")
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_by_image(tmp_path):
    port = _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_worker, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    for p in procs:
        if p.is_alive():
            p.kill()
            pytest.fail("gloo rank did not finish")
        assert p.exitcode == 0
    assert (tmp_path / "ok").read_text() == "1"
