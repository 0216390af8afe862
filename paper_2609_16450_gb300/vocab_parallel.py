"""Vocabulary-parallel LM head across GPUs: the plumbing around
ebd_lm_shard_state and ebd_merge_shard_states (every step of the arithmetic
runs in libebd.so).

Each rank holds the rows [v0, v1) of W_lm given by shard_range, reduces them
to one 32-byte softmax state per window row (ebd_lm_shard_state), the states
of all ranks are all-gathered with torch.distributed (NCCL between GPUs),
and every rank merges them into the statistics of the whole vocabulary
(ebd_merge_shard_states); the decision (ebd_decide) then runs on every rank
on identical inputs.  The statistics are those of App. B (Eq.
app-confidence), Sec. 5.1 and Sec. 5.2; the merge of range states is
associative, so any partition of the vocabulary gives the same statistics up
to the rounding of the merge order.
"""
from __future__ import annotations

from typing import Optional, Tuple

import torch
import torch.distributed as dist

from . import _ebd as E

STATE_WORDS = 8  # m, S, T, l2, idx (int32 bits), three zero words
UNIT = 64        # vocabulary rows of one LM-head work unit; shards start on a unit


def shard_range(vocab: int, world: int, rank: int) -> Tuple[int, int]:
    """Rows [v0, v1) of W_lm held by `rank` of `world`: the 64-row units of
    the vocabulary split into contiguous, nearly equal runs."""
    if not 0 <= rank < world:
        raise ValueError("rank out of range")
    units = (vocab + UNIT - 1) // UNIT
    u0 = rank * units // world
    u1 = (rank + 1) * units // world
    return min(vocab, u0 * UNIT), min(vocab, u1 * UNIT)


def shard_weights(w_lm: torch.Tensor, vocab: int, d_model: int, v0: int, v1: int,
                  layout: int) -> torch.Tensor:
    """This rank's rows [v0, v1) of W_lm as a contiguous tensor: a row slice
    of the row-major [vocab][d_model] matrix (layout 0), or the run of tiles
    of the tiled copy of ebd_pack_lm_head (layout 1), which holds whole
    64-row units; v0 must be a multiple of 64."""
    if v0 % UNIT:
        raise ValueError("a shard starts on a 64-row unit")
    if layout == 0:
        return w_lm.view(vocab, d_model)[v0:v1]
    nkb = (d_model + 63) // 64
    tile = nkb * 64 * 64  # elements of one unit's tiles
    flat = w_lm.view(-1)
    return flat[(v0 // UNIT) * tile:((v1 + UNIT - 1) // UNIT) * tile]


def new_state(rows: int, device) -> torch.Tensor:
    return torch.empty((max(rows, 1), STATE_WORDS), dtype=torch.float32, device=device)


def gather_states(state: torch.Tensor, group=None) -> torch.Tensor:
    """All-gather of every rank's [rows][8] states into [world][rows][8], in
    rank order (any order merges to the same statistics)."""
    world = dist.get_world_size(group)
    out = torch.empty((world,) + tuple(state.shape), dtype=state.dtype, device=state.device)
    if state.is_cuda:
        dist.all_gather_into_tensor(out, state.contiguous(), group=group)
    else:
        dist.all_gather(list(out.unbind(0)), state.contiguous(), group=group)
    return out


def lm_stats(handle, args: "E.ebd_step_args", w_shard: torch.Tensor, v0: int, v1: int,
             group=None, stream: Optional[int] = None) -> torch.Tensor:
    """Step 2 of the step, sharded: this rank's state from w_shard (its rows
    [v0, v1) of W_lm, in args.w_lm_layout), all-gathered, merged into
    args.conf/entropy/ent_norm/gap/argmax.  Returns the gathered states.
    The library calls and the collective are ordered on torch's current
    stream (`stream` must be that stream's handle, or None for it)."""
    s = torch.cuda.current_stream().cuda_stream if stream is None else stream
    state = new_state(args.rows, w_shard.device)
    args.w_lm = w_shard.data_ptr()
    E.check(E.ebd_lm_shard_state(handle.h, args, v0, v1 - v0, state.data_ptr(), s), handle.h)
    states = gather_states(state[:args.rows], group)
    E.check(E.ebd_merge_shard_states(handle.h, states.data_ptr(), states.shape[0], args, s),
            handle.h)
    return states
