"""One MCA chain whose samples are split over ranks (one process per GPU).

The training loss is a sum over samples (Eq. 2), so the loss change of a proposal is the sum of its
changes on disjoint sample shards. Each rank holds one handle on its own samples. Per batch of
trials every rank

  1. draws the batch's proposals and evaluates them on its shard, without committing
     (mca_eval_trials: the same Philox proposals and kernels as mca_run);
  2. exchanges the K partial loss changes with the other ranks (one all-gather of K fp64 values
     through torch.distributed: NCCL between GPUs, gloo on CPU ranks) and adds them in rank order,
     so every rank holds bit-identical sums;
  3. takes the batch's decision from the sums (mca_decide_batch: the lowest-index trial with
     dS <= theta, Eq. 6, or Eq. 7 with theta from the trial's own Philox word and the chain's whole
     sample count) -- the same decision on every rank;
  4. commits it on its own shard (mca_force_decisions for the consumed trials, then mca_run over
     them: the shard's kernels re-evaluate those candidates and take the given decisions).

No device work waits for another rank; the exchange is the only collective. The batch width
follows the observed acceptance rate (ceil(c / p) trials, p = (A + 1/2) / (T + 1) from counts
decayed by 0.95 per batch, at most K); every rank computes it from the same decisions.

A shard is any object with eval_trials / decide / commit (LibraryShard wraps a handle), so the
same chain runs over other evaluators, e.g. in CPU tests.
"""
from __future__ import annotations

import math
from typing import Dict, Optional

import numpy as np

RATE_DECAY = 0.95


class LibraryShard:
    """A rank's shard: an mca handle created on the rank's samples (mca.mca_create or
    mca.create_from_workload on the shard's rows)."""

    def __init__(self, handle):
        from . import mca
        self.mca = mca
        self.h = handle

    def eval_trials(self, seed: int, tau: int, n: int):
        """(valid [n] bool, partial dS [n] float64 with 0 for invalid trials, flat idx [n])."""
        rec = self.mca.mca_eval_trials(self.h, seed, tau, n)
        valid = rec["valid"].astype(bool)
        return valid, np.where(valid, rec["dS"], 0.0), rec["idx"].astype(np.int64)

    def decide(self, seed: int, tau: int, valid, dS, n_samples: int) -> int:
        return self.mca.mca_decide_batch(self.h, seed, tau, valid, dS, n_samples)

    def commit(self, seed: int, tau: int, m: int, kstar: int):
        acc = np.zeros(m, np.uint8)
        if kstar >= 0:
            acc[kstar] = 1
        self.mca.mca_force_decisions(self.h, np.arange(tau, tau + m, dtype=np.uint64), acc)
        st = self.mca.mca_run(self.h, m, seed)
        self.mca.mca_force_decisions(self.h, [], [])
        return st


def batch_width(acc: float, trials: float, c: float, K: int) -> int:
    p = (acc + 0.5) / (trials + 1.0)
    w = math.ceil(c / p)
    return max(1, min(K, w))


class ShardedChain:
    """Drives one chain over the ranks of a torch.distributed group (or a single process when no
    group is initialised). n_samples: the chain's whole sample count (Eq. 7's N)."""

    def __init__(self, shard, n_samples: int, K: int = 64, c: float = 1.0, group=None):
        self.shard = shard
        self.n_samples = int(n_samples)
        self.K = int(K)
        self.c = float(c)
        self.group = group
        self.tau = 0
        self.rate_acc = 0.0
        self.rate_trials = 0.0
        self.stats = {"trials": 0, "accepts": 0, "batches": 0, "exchanges": 0}

    def _world(self):
        import torch.distributed as dist
        if dist.is_available() and dist.is_initialized():
            return dist.get_world_size(self.group)
        return 1

    def exchange(self, part: np.ndarray) -> np.ndarray:
        """All-gather every rank's partial loss changes and add them in rank order."""
        if self._world() == 1:
            return part.astype(np.float64)
        import torch
        import torch.distributed as dist
        dev = torch.device("cpu")
        if dist.get_backend(self.group) == "nccl":
            dev = torch.device("cuda", torch.cuda.current_device())
        t = torch.from_numpy(np.ascontiguousarray(part, np.float64)).to(dev)
        out = [torch.empty_like(t) for _ in range(self._world())]
        dist.all_gather(out, t, group=self.group)
        self.stats["exchanges"] += 1
        total = np.zeros(len(part), np.float64)
        for g in out:                                # rank order: the same sums on every rank
            total = total + g.cpu().numpy()
        return total

    def run(self, n_trials: int, seed: int, forced: Optional[Dict[int, bool]] = None) -> dict:
        """Run n_trials trials from the chain's counter. forced: {tau: accept} decisions taken in
        place of the rule (a test hook, as mca_force_decisions)."""
        end = self.tau + int(n_trials)
        while self.tau < end:
            tau = self.tau
            kb = min(batch_width(self.rate_acc, self.rate_trials, self.c, self.K), end - tau)
            valid, part, _ = self.shard.eval_trials(seed, tau, kb)
            dS = self.exchange(part)
            kstar = self._decide(seed, tau, valid, dS, forced)
            m = kstar + 1 if kstar >= 0 else kb
            self.shard.commit(seed, tau, m, kstar)
            acc = 1 if kstar >= 0 else 0
            self.rate_acc = self.rate_acc * RATE_DECAY + acc
            self.rate_trials = self.rate_trials * RATE_DECAY + m
            self.tau += m
            self.stats["trials"] += m
            self.stats["accepts"] += acc
            self.stats["batches"] += 1
        return dict(self.stats, tau=self.tau)

    def _decide(self, seed, tau, valid, dS, forced) -> int:
        kb = len(valid)
        if not forced or not any((tau + k) in forced for k in range(kb)):
            return self.shard.decide(seed, tau, valid, dS, self.n_samples)
        for k in range(kb):
            if (tau + k) in forced:
                if forced[tau + k]:
                    return k
            elif self.shard.decide(seed, tau + k, valid[k:k + 1], dS[k:k + 1],
                                   self.n_samples) == 0:
                return k
        return -1
