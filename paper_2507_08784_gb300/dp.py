"""Data-parallel GreedyLore across processes: Algorithm 3's All-Reduce lines made explicit.

Each rank owns a shard of the N nodes of a data-parallel group (the same shard size on every
rank).  A step runs in three phases of a per-shard engine; between them the buffers the engine
exposes are averaged over the ranks with torch.distributed all-reduces, in place:

* begin(G)   the shard's composed gradients M_i = G_i + E_i; exposes the shard's Approx-Top-r
             scores lambda-bar (m' floats, Algorithm 2) or, on a refresh / warm-up step, the
             shard's node mean Mbar (m' x n' floats);
* select()   the refresh of the averaged Mbar (Eq. SVD-P1) or the arg-top-r of the averaged
             lambda-bar, P = U[:, J], and the shard's projected mean Rbar (r x n' floats);
* finish(X)  Ghat = P Rbar with the averaged Rbar (or Mbar), the optimizer on X, and the error
             feedback of the shard's nodes.

The floats exchanged are Table 2's: m' + r n' on a compressed step and m' n' on an Algorithm 3
refresh (``floats_exchanged`` counts them).  ``ShardEngine`` runs the phases on this rank's GPU
through the C ABI (glr_dp_begin / glr_dp_select / glr_dp_finish).
"""
from __future__ import annotations

from typing import Callable, List, Optional, Sequence

import torch

from . import GreedyLore, glr_dp_begin, glr_dp_finish, glr_dp_select


class _DeviceArray:
    """A float32 device buffer of the library's state seen through the CUDA array interface."""

    def __init__(self, ptr: int, floats: int):
        self.__cuda_array_interface__ = {"shape": (floats,), "typestr": "<f4", "data": (ptr, False),
                                         "version": 3, "strides": None}


def device_view(ptr: int, floats: int) -> torch.Tensor:
    """A torch view (no copy) of `floats` float32 values at device address `ptr`."""
    return torch.as_tensor(_DeviceArray(ptr, floats), device="cuda")


class ShardEngine:
    """The three phases of a step for this rank's shard, on its GPU (a GreedyLore handle created
    with the shard's node count)."""

    def __init__(self, layer: GreedyLore, stream=None):
        self.layer, self.stream = layer, stream

    def begin(self, G: Sequence[torch.Tensor]) -> List[torch.Tensor]:
        return [device_view(p, n) for p, n in glr_dp_begin(self.layer.handle, G, self.stream)]

    def select(self) -> List[torch.Tensor]:
        return [device_view(p, n) for p, n in glr_dp_select(self.layer.handle, self.stream)]

    def finish(self, X: torch.Tensor) -> None:
        glr_dp_finish(self.layer.handle, X, self.stream)


def allreduce_mean(group=None) -> Callable[[torch.Tensor], None]:
    """The exchange over a torch.distributed group: in-place all-reduce of the sum, divided by the
    group's size."""
    import torch.distributed as dist

    world = dist.get_world_size(group)

    def average(buf: torch.Tensor) -> None:
        dist.all_reduce(buf, op=dist.ReduceOp.SUM, group=group)
        buf.div_(world)
    return average


class DataParallelGreedyLore:
    """One layer matrix's GreedyLore step over the ranks of a data-parallel group.

    engine: an object with begin(G), select() and finish(X) (``ShardEngine`` for the GPU library);
    average: the in-place exchange of one buffer (``allreduce_mean(group)``; None: a single rank).
    """

    def __init__(self, engine, average: Optional[Callable[[torch.Tensor], None]] = None):
        self.engine, self.average = engine, average
        self.floats_exchanged = 0            # over all steps, per rank (Table 2's per-node count)
        self.last_step_floats = 0

    def _exchange(self, bufs: List[torch.Tensor]) -> None:
        for b in bufs:
            self.last_step_floats += b.numel()
            if self.average is not None:
                self.average(b)

    def step(self, G: Sequence[torch.Tensor], X: torch.Tensor) -> None:
        self.last_step_floats = 0
        self._exchange(self.engine.begin(G))
        self._exchange(self.engine.select())
        self.engine.finish(X)
        self.floats_exchanged += self.last_step_floats
