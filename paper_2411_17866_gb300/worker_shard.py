"""Worker-sharded rounds of Algorithm 1: the n workers split over G processes (host-side logic).

In the paper's deployment every worker is a device (Sec. 5 trains GPT-2 on 8 and 16 GPUs) and
Algorithm 1's all-reduce averages the workers' models once per round.  Here rank r of G holds a
contiguous group of the workers (their models x_i and base-optimizer states) and runs their tau local
steps; the round's global step is computed in parameter shards: the model is cut into G contiguous
ranges (shard.shard_bounds), rank s owns range s, keeps the global momentum m of that range only (the
layered, ZeRO-style placement that Sec. 3 sketches for a distributed optimizer) and computes the global
step there.

One round, on every rank:
  1. the tau local steps of the rank's workers (the compute backend);
  2. an all-to-all: every rank sends each owner its workers' models on the owner's range, so that the
     owner holds all n models of its range, in worker order 0..n-1 (the groups are contiguous and in
     rank order, so the ranks' blocks arrive in worker order);
  3. the owner's global step on its range: Delta = (1/n) sum_{i=0..n-1} (x - x_i), summed in worker
     order, then Eqs. (ut-update), (model-update), (mom-update) and the randomized sign keyed by the
     range's place in the whole model (the compute backend);
  4. an all-gather of the new x, from which every rank's workers start the next round (the backend).

Why an all-to-all of the models rather than a reduce-scatter of the differences: a reduce-scatter adds
the ranks' partial sums in the collective's own order, so Delta would differ from the one-process sum
in its last bits; with the models exchanged the owner adds the n differences in the fixed order, and
the G processes compute bit for bit what one process computes.  With one worker per rank (n = G, the
paper's setting) both move the same bytes: (G - 1)/G of d values per rank and round, plus the same
again for the all-gather.

The compute backend is an object with
  local_steps(t)                    the tau local steps of round t for the rank's workers;
  replicas() -> [n_r, d] tensor     the rank's workers' models after them (fp32, the collective's device);
  global_step(shard, X_shard, t) -> (x_shard, piece_stats)
                                    the global step on the owned range, from the n models of that range
                                    ([n, count] tensor); returns the range's new x and the statistics of
                                    the shard's pieces (or None);
  restart(x)                        the new global model x (all d values): every worker starts from it.
Two backends exist: the oracle's (tests/test_worker_shard.py) and LibraryWorkers below, which runs the
rank's workers and the owner's global step in the library on the process's GPU.
This module holds no arithmetic of the method; it places the workers and the ranges, and moves data.
"""
from __future__ import annotations

import dataclasses

from . import shard as S


@dataclasses.dataclass(frozen=True)
class WorkerGroup:
    rank: int
    world: int
    n: int               # workers in all
    first_worker: int    # global index of the rank's first worker
    count: int           # workers of the rank


def worker_groups(n: int, world: int):
    """Contiguous groups of the n workers over `world` ranks, in rank order, as equal as possible."""
    if world < 1 or n < world:
        raise ValueError("every rank needs at least one worker (n >= world >= 1)")
    cuts = [r * n // world for r in range(world)] + [n]
    return [WorkerGroup(r, world, n, cuts[r], cuts[r + 1] - cuts[r]) for r in range(world)]


class WorkerShardedRound:
    """Drives the rounds of one rank.  tensors: the whole model's tensor list; backend: see the module
    docstring; group: a torch.distributed process group (None: the default group)."""

    def __init__(self, tensors, n: int, backend, group=None, align: int = 64):
        import torch.distributed as dist
        self.group = group
        self.world = dist.get_world_size(group)
        self.rank = dist.get_rank(group)
        self.tensors = list(tensors)
        self.d = sum(int(t.numel) for t in self.tensors)
        self.groups = worker_groups(n, self.world)
        self.workers = self.groups[self.rank]
        self.bounds = S.shard_bounds(self.d, self.world, align)
        self.shard = S.shard_layout(self.tensors, self.world, self.rank, align)
        self.backend = backend
        self.t = 0

    def exchange(self, X_local):
        """Step 2: every owner receives the n models of its range, rows in worker order ([n, count])."""
        import torch
        import torch.distributed as dist
        n_r = X_local.shape[0]
        send = torch.cat([X_local[:, a:b].reshape(-1) for a, b in self.bounds])
        send_splits = [n_r * (b - a) for a, b in self.bounds]
        recv_splits = [g.count * self.shard.count for g in self.groups]
        recv = torch.empty(sum(recv_splits), dtype=X_local.dtype, device=X_local.device)
        dist.all_to_all_single(recv, send, recv_splits, send_splits, group=self.group)
        return recv.view(self.workers.n, self.shard.count)

    def gather_x(self, x_shard):
        """Step 4: the new x, all d values, on every rank (ranges padded to the longest for the all-gather)."""
        import torch
        import torch.distributed as dist
        longest = max(b - a for a, b in self.bounds)
        padded = torch.zeros(longest, dtype=x_shard.dtype, device=x_shard.device)
        padded[:x_shard.numel()] = x_shard
        parts = [torch.empty_like(padded) for _ in range(self.world)]
        dist.all_gather(parts, padded, group=self.group)
        return torch.cat([p[:b - a] for p, (a, b) in zip(parts, self.bounds)])

    def run_round(self, with_stats: bool = False):
        """One round of Algorithm 1 over all ranks; with_stats: the whole model's per-tensor statistics
        (summed over the ranges' pieces on every rank), else None."""
        self.backend.local_steps(self.t)
        X_shard = self.exchange(self.backend.replicas())
        x_shard, piece_stats = self.backend.global_step(self.shard, X_shard, self.t)
        x = self.gather_x(x_shard)
        self.backend.restart(x)
        self.t += 1
        if not with_stats:
            return None
        mine = S.stats_by_tensor(self.shard, piece_stats, len(self.tensors))
        return S.all_reduce_stats(mine)


class LibraryWorkers:
    """The compute backend on this process's CUDA device, through the library's C ABI.

    - The rank's workers are one handle of group.count workers over the whole model, placed at
      group.first_worker (dsm_set_first_worker), so that they draw the synthetic gradients of those
      workers of the n.
    - The owned range's global step is dsm_global_step_noalloc on the owner's x and m of the range and
      the n models of the range (Algorithm 1's global step, or the SlowMo, signed SlowMo and Lookahead
      variants that entry point also runs), with the range's layout placed at its first element
      (dsm_layout.first_element: the randomized sign's counters are those of the whole model).
    - The restart is dsm_end_round with the gathered x: the handle's workers start the next round from
      it, their base-optimizer states carry over.
    comm_device: where the collectives' tensors live ("cpu" for gloo, the CUDA device for NCCL)."""

    def __init__(self, tensors, n: int, tau: int, hp, group: WorkerGroup, shard: S.Shard, device="cuda",
                 comm_device="cpu"):
        import torch
        from . import dsm
        self._dsm = dsm
        self.tau, self.n = tau, n
        self.device = torch.device(device)
        self.comm = torch.device(comm_device)
        self.run = dsm.DistributedSignMomentum(tensors, group.count, tau, hp, device=self.device)
        self.run.set_first_worker(group.first_worker)
        self.shard = shard
        self.layout = dsm.make_layout(shard.tensors, first_element=shard.first_element)
        self.hparams = dsm.make_hparams(hp)
        # the owner's state of its range: x, m (m_0 = 0) and the n models, rows padded to a multiple of 8
        self.stride = max(8, -(-shard.count // 8) * 8)
        self.m = torch.zeros(max(shard.count, 1), dtype=torch.float32, device=self.device)
        self.x = torch.empty(max(shard.count, 1), dtype=torch.float32, device=self.device)
        self.X = torch.empty((n, self.stride), dtype=torch.float32, device=self.device)

    def local_steps(self, t):
        for k in range(self.tau):
            self.run.fill_synthetic_grads(t * self.tau + k)
            self.run.local_step()

    def replicas(self):
        import torch
        if self.comm.type == "cuda":
            return torch.stack([self.run.replica_view(i) for i in range(self.run.n)])
        return torch.stack([self.run.read(self._dsm.BUF_REPLICA, i) for i in range(self.run.n)])

    def global_step(self, shard, X_shard, t):
        import torch
        dsm = self._dsm
        count = shard.count
        if count == 0:
            return torch.empty(0, dtype=torch.float32, device=self.comm), []
        with torch.cuda.device(self.device):
            self.X[:, :count].copy_(X_shard.to(self.device))
            self.run.read(dsm.BUF_X, offset=shard.first_element, count=count, out=self.x[:count])
            stats = (dsm.dsm_tensor_stats * len(shard.pieces))()
            dsm.dsm_global_step_noalloc(self.layout, self.n, self.hparams, self.run.info().gamma, t,
                                        self.x.data_ptr(), self.m.data_ptr(), self.X.data_ptr(), self.stride,
                                        stats)
            return self.x[:count].to(self.comm), [s.as_dict() for s in stats]

    def restart(self, x):
        import torch
        with torch.cuda.device(self.device):
            self.run.end_round(x)

    def momentum(self):
        """The owner's global momentum of its range (CPU)."""
        return self.m[:self.shard.count].cpu()
