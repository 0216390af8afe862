"""The vocabulary-parallel LM head's host logic on CPU, as two and three gloo
ranks (127.0.0.1): the shard ranges partition the vocabulary on 64-row units,
and the all-gather of the per-rank states (product code,
vocab_parallel.gather_states, in the library's 8-word state layout) merges
into the statistics of the whole vocabulary.  Each rank's state is the
oracle's range state of its shard (the GPU computes it in ebd_lm_shard_state,
tested by tests/test_gpu_vocab_parallel.py)."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import ebd_oracle as o
from paper_2609_16450_gb300 import vocab_parallel as vp

V, ROWS = 1000, 6


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _logits():
    rng = np.random.default_rng(77)
    L = rng.standard_normal((ROWS, V)) * np.array([[0.5], [2], [6], [12], [1], [3]])
    L[5, 70] = L[5, 900] = L[5].max() + 2.0  # equal maxima on two ranks
    return L


def _pack(st: "o.RangeState") -> torch.Tensor:
    t = torch.zeros((ROWS, vp.STATE_WORDS), dtype=torch.float32)
    t[:, 0] = torch.from_numpy(st.m.astype(np.float32))
    t[:, 1] = torch.from_numpy(st.S.astype(np.float32))
    t[:, 2] = torch.from_numpy(st.T.astype(np.float32))
    t[:, 3] = torch.from_numpy(st.l2.astype(np.float32))
    t[:, 4] = torch.from_numpy(st.idx.astype(np.int32)).view(torch.float32)
    return t


def _unpack(t: torch.Tensor) -> "o.RangeState":
    a = t.numpy()
    return o.RangeState(m=a[:, 0].astype(np.float64), S=a[:, 1].astype(np.float64),
                        T=a[:, 2].astype(np.float64), l2=a[:, 3].astype(np.float64),
                        idx=a[:, 4].copy().view(np.int32).astype(np.int64))


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        L = _logits()
        v0, v1 = vp.shard_range(V, world, rank)
        mine = _pack(o.range_state(L[:, v0:v1], v0))
        gathered = vp.gather_states(mine)
        out[rank] = (v0, v1, gathered.numpy().copy())
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_gathered_shard_states_merge_to_the_whole_vocabulary(world):
    import torch.multiprocessing as mp
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    ranges = [out[r][:2] for r in range(world)]
    assert ranges[0][0] == 0 and ranges[-1][1] == V
    for (a, b), (c, d) in zip(ranges[:-1], ranges[1:]):
        assert b == c and a % 64 == 0
    # every rank gathered the same states, in rank order
    for r in range(1, world):
        np.testing.assert_array_equal(out[r][2], out[0][2])
    L = _logits()
    states = [_unpack(torch.from_numpy(out[0][2][g])) for g in range(world)]
    st = o.merge_range_states(states, V)
    ref = o.softmax_stats(L)
    for k in ("conf", "entropy", "ent_norm", "gap"):
        np.testing.assert_allclose(getattr(st, k), getattr(ref, k), rtol=1e-5, atol=1e-6, err_msg=k)
    assert st.argmax.tolist() == ref.argmax.tolist()
    assert st.argmax[5] == 70


def test_shard_ranges_cover_the_vocabulary():
    for vocab in (64, 1000, 126464, 152064):
        for world in (1, 2, 3, 8):
            rs = [vp.shard_range(vocab, world, r) for r in range(world)]
            assert rs[0][0] == 0 and rs[-1][1] == vocab
            assert all(b == c for (_, b), (c, _) in zip(rs[:-1], rs[1:]))
            assert all(a % 64 == 0 for a, _ in rs)
