"""The N > 1 path on the CPU with gloo (world size 2): bench.py's max-over-ranks timing and
summed kept tokens, per-rank batches, and the data-parallel reading of the loss denominator
(each rank passing the global kept-token count gives per-rank losses that sum to the loss of
one process over the concatenated batch)."""
import os
import socket

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import oracle
    from paper_2609_36932_gb300 import workloads
    # 1. timing reduction: max of the times, sum of the kept tokens
    ms, kept = bench.combine_ranks(10.0 + 5 * rank, 100 + rank, world, torch.device("cpu"))
    # 2. this rank's batch and its oracle loss with the global kept-token denominator
    w = workloads.get("tiny")
    b = workloads.make_batch(w, bench.rank_seed(0, rank))
    adv, _ = oracle.advantage(b["rewards"], w.G)
    keep, _ = oracle.prune(b["rewards"], b["ids"], b["off"], w.G, 1, w.tau, w.keep_cap, 1)
    comp = oracle.compact(keep, b["off"])
    tk = torch.tensor([comp["T_kept"]], dtype=torch.int64)
    dist.all_reduce(tk)
    rng = np.random.default_rng(rank)
    logits = rng.standard_normal((b["T"], w.V)).astype(np.float32)
    old = rng.standard_normal(b["T"]).astype(np.float32) - 7.0
    ref = old + 0.1
    r = oracle.loss(logits, w.V, b["ids"], old, ref, adv, comp["token_rollout"],
                    row_index=comp["src_token"], denom_tokens=int(tk.item()), want_dlogits=False)
    loss = torch.tensor([r["loss"]], dtype=torch.float64)
    dist.all_reduce(loss)
    out[rank] = dict(ms=ms, kept=kept, global_tk=int(tk.item()), loss_sum=float(loss.item()),
                     ids_head=b["ids"][:8].tolist())
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks():
    import torch.multiprocessing as mp
    mgr = mp.Manager()
    out = mgr.dict()
    port = free_port()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    a, b = out[0], out[1]
    assert a["ms"] == b["ms"] == 15.0 and a["kept"] == b["kept"] == 201.0
    assert a["ids_head"] != b["ids_head"]  # each rank its own batch
    assert a["loss_sum"] == b["loss_sum"]
    # one process over both batches, one denominator
    import oracle
    from paper_2609_36932_gb300 import workloads
    import bench
    w = workloads.get("tiny")
    total, tk_all = 0.0, 0
    parts = []
    for rank in range(2):
        bb = workloads.make_batch(w, bench.rank_seed(0, rank))
        adv, _ = oracle.advantage(bb["rewards"], w.G)
        keep, _ = oracle.prune(bb["rewards"], bb["ids"], bb["off"], w.G, 1, w.tau, w.keep_cap, 1)
        comp = oracle.compact(keep, bb["off"])
        tk_all += comp["T_kept"]
        parts.append((bb, adv, comp, rank))
    assert tk_all == a["global_tk"]
    for bb, adv, comp, rank in parts:
        rng = np.random.default_rng(rank)
        logits = rng.standard_normal((bb["T"], w.V)).astype(np.float32)
        old = rng.standard_normal(bb["T"]).astype(np.float32) - 7.0
        ref = old + 0.1
        total += oracle.loss(logits, w.V, bb["ids"], old, ref, adv, comp["token_rollout"],
                             row_index=comp["src_token"], denom_tokens=tk_all,
                             want_dlogits=False)["loss"]
    assert a["loss_sum"] == pytest.approx(total, rel=1e-12)
