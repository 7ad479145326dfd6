"""Complete-prefix shadow evaluation batched into the rollout's packed forward
(App. B.2 "Shadow evaluation procedure").

For each image the rollout prunes at its pruning blocks.  The shadow of
prefix l replays the rollout's deletions at blocks 0..l and runs every later
block unpruned; the empty prefix is the Native forward.  A shadow is identical
to the rollout up to and including block l, so it is branched off the
rollout's output of block l (``dora_branch``: the image's surviving rows
copied as a new sequence of the same packed batch) and from then on rides in
the same kernels as the rollout with its keep count equal to its length.  The
Native copies are branched just before the first pruning block (until then
the rollout is the Native forward, so those blocks run once); no shadow is
branched at the last pruning block, whose prefix is the rollout itself.  Every GEMM row and every
attention sequence is computed independently of the others in the batch, so
a shadow computed here has the same bits as the same prefix run alone.

All arithmetic runs in libdora's kernels; this module only orders the calls
and owns the buffers.
"""
from __future__ import annotations

import contextlib

import torch

from . import (alloc_workspace, dora_branch, dora_classifier_head, dora_classifier_head_lc1,
               dora_gather_scores, dora_kd_cost, dora_pl_logprob, dora_pl_sample,
               dora_pruned_block, dora_step_rewards)


class ShadowRollout:
    """Buffers for a batch of ``batch`` images of ``n_tokens`` rows each, a
    depth-``len(blocks)`` forward pruned at ``prune_blocks``, with Native and
    complete-prefix shadows riding along."""

    def __init__(self, blocks: list, batch: int, n_tokens: int, prune_blocks, device,
                 classes: int = 1000):
        if not prune_blocks or list(prune_blocks) != sorted(set(prune_blocks)) or \
                prune_blocks[-1] >= len(blocks) or prune_blocks[0] < 0:
            raise ValueError("prune_blocks must be increasing block indices, at least one")
        self.blocks = blocks
        self.b = batch
        self.n_tokens = n_tokens
        self.prune = list(prune_blocks)
        self.branch_at = self.prune[:-1]
        self.depth = len(blocks)
        self.dim = blocks[0].dim
        self.nseq = batch * (2 + len(self.branch_at))
        self.t_cap = batch * n_tokens * (2 + len(self.branch_at))
        d, t, dev = self.dim, self.t_cap, device
        self.x = [torch.zeros(t, d, dtype=torch.bfloat16, device=dev) for _ in range(2)]
        self.mv = [torch.zeros(t, 2, dtype=torch.float32, device=dev) for _ in range(2)]
        self.ids = [torch.zeros(t, dtype=torch.int32, device=dev) for _ in range(2)]
        self.cu = [torch.zeros(self.nseq + 1, dtype=torch.int32, device=dev) for _ in range(2)]
        self.keep = torch.zeros(self.nseq, dtype=torch.int32, device=dev)
        self.scores = torch.zeros(t, dtype=torch.float32, device=dev)
        self.kept = torch.zeros(t, dtype=torch.int32, device=dev)
        self.src = torch.arange(batch, dtype=torch.int32, device=dev)
        self.ws = alloc_workspace(t, self.nseq, blocks[0], dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.classes_pad = (classes + 31) // 32 * 32
        self.classes = classes
        self.logits = torch.zeros(self.nseq, self.classes_pad, dtype=torch.bfloat16, device=dev)
        self.cost = torch.zeros(self.nseq, dtype=torch.float32, device=dev)
        # every sequence compares with its image's Native logits
        self.image_of = torch.arange(self.nseq, dtype=torch.int32, device=dev) % batch
        self.head_ws = None
        # training rollouts (App. A.3): per pruning block the selector scores,
        # the rollout's boundaries, the sampled removal order and its
        # log-probability
        npb = len(self.prune)
        self.k_cap = n_tokens - 1
        self.keys = torch.zeros(t, dtype=torch.float32, device=dev)
        self.gum = torch.zeros(batch * n_tokens, dtype=torch.float32, device=dev)
        self.s_hist = [torch.zeros(batch * n_tokens, dtype=torch.float32, device=dev)
                       for _ in range(npb)]
        self.cu_hist = [torch.zeros(batch + 1, dtype=torch.int32, device=dev) for _ in range(npb)]
        self.order = torch.full((npb, batch, self.k_cap), -1, dtype=torch.int32, device=dev)
        self.logp = torch.zeros(npb, batch, dtype=torch.float32, device=dev)
        self.grad = [torch.zeros(batch * n_tokens, dtype=torch.float32, device=dev)
                     for _ in range(npb)]
        # sequence layout after the forward: rollout, Native, then one group
        # of `batch` shadows per branching block
        self.groups = {"rollout": 0, "native": batch}
        for j, l in enumerate(self.branch_at):
            self.groups[l] = batch * (2 + j)

    def launches(self) -> int:
        """Kernel launches of one forward() without the head (for reporting)."""
        n = 2                                           # Native branch: scan + copy
        for l in range(self.depth):
            n += 6 + (l == 0) + (l + 1 < self.depth)
            if l in self.prune:
                n += 3                                  # gather, select, compact
                if l in self.branch_at:
                    n += 2
        return n

    def forward(self, x0, cu0, ids0, tables, keeps, stream=None, stop=None, gumbel=None,
                removals=None):
        """Rollout + Native + shadows through every block.  x0 bf16 [B N, d],
        cu0 int32 [B + 1], ids0 int32 [B N]; tables[j] fp32 [B, stride]
        deletion-score tables keyed by original token id and keeps[j] int32
        [B] keep counts for pruning block j.  A training rollout also passes
        gumbel[j] (fp32 [B, stride] standard Gumbel noise keyed, like the
        scores, by original token id) and removals[j] (int32 [B], k = rows -
        keep counts): the removal order
        is then sampled (dora_pl_sample) and the block deletes the sampled set
        by taking the perturbed keys as its scores.  Returns (x, cu, ids) of the whole
        packed batch (sequence order: rollout, Native, shadow groups).  With
        ``stop`` the batch is returned after the first ``stop`` blocks (and
        their branches)."""
        with torch.cuda.stream(stream) if stream is not None else contextlib.nullcontext():
            return self._forward(x0, cu0, ids0, tables, keeps, stream,
                                 self.depth if stop is None else stop, gumbel, removals)

    def _forward(self, x0, cu0, ids0, tables, keeps, stream, stop, gumbel, removals):
        b = self.b
        rows = x0.shape[0]
        x, mv, ids = self.x[0], None, self.ids[0]
        x[:rows].copy_(x0)
        ids[:rows].copy_(ids0)
        cu = self.cu[0]
        cu[:b + 1].copy_(cu0)
        nseq, p, q = b, 0, 0
        for l, w in enumerate(self.blocks[:stop]):
            out = self.x[1 - p]
            mv_out = self.mv[1 - p] if l + 1 < self.depth else None
            if l == self.prune[0]:
                # Native copies: whole images, never pruned from here on
                dora_branch(x, cu[:b + 1], self.src, cu[:2 * b + 1], ids=ids, x_moments=mv,
                            len_out=self.keep[b:2 * b], status=self.status, stream=stream)
                nseq = 2 * b
            if l in self.prune:
                j = self.prune.index(l)
                self.keep[:b].copy_(keeps[j])
                sc = self.scores
                if gumbel is not None:
                    sj = self.s_hist[j]
                    dora_gather_scores(tables[j], ids, cu[:b + 1], sj, status=self.status,
                                       stream=stream)
                    dora_gather_scores(gumbel[j], ids, cu[:b + 1], self.gum, status=self.status,
                                       stream=stream)
                    self.cu_hist[j].copy_(cu[:b + 1])
                    dora_pl_sample(sj, self.gum, self.cu_hist[j], removals[j], self.order[j],
                                   keys_out=self.keys, status=self.status, stream=stream)
                    sc = self.keys
                else:
                    dora_gather_scores(tables[j], ids, cu[:b + 1], sc, status=self.status,
                                       stream=stream)
                cu_out, idn = self.cu[1 - q], self.ids[1 - q]
                dora_pruned_block(x, cu[:nseq + 1], w, self.n_tokens, out, self.ws, ids_in=ids,
                                  scores=sc, keep_counts=self.keep[:nseq],
                                  cu_out=cu_out[:nseq + 1], ids_out=idn, kept_idx=self.kept,
                                  x_in_moments=mv, x_out_moments=mv_out, stream=stream)
                if l in self.branch_at:
                    dora_branch(out, cu_out[:nseq + 1], self.src, cu_out[:nseq + b + 1], ids=idn,
                                x_moments=mv_out, len_out=self.keep[nseq:nseq + b],
                                status=self.status, stream=stream)
                    nseq += b
                cu, q, ids = cu_out, 1 - q, idn
            else:
                dora_pruned_block(x, cu[:nseq + 1], w, self.n_tokens, out, self.ws, ids_in=ids,
                                  x_in_moments=mv, x_out_moments=mv_out, stream=stream)
            x, mv, p = out, mv_out, 1 - p
        self.nseq_out = nseq
        return x, cu[:nseq + 1], ids

    def logprob(self, removals, dlogp=None, stream=None):
        """Plackett-Luce log-probabilities [pruning blocks, B] of the sampled
        removal orders of the last training forward, and their gradients with
        respect to the selector scores (times dlogp [B], e.g. advantages)."""
        for j in range(len(self.prune)):
            dora_pl_logprob(self.s_hist[j], self.cu_hist[j], removals[j], self.order[j],
                            self.logp[j], grad=self.grad[j], dlogp=dlogp, status=self.status,
                            stream=stream)
        return self.logp, self.grad

    def rewards(self, removals, a, reward, ret=None, stream=None):
        """Local rewards [P, B] of the last training forward's actions from the
        fidelity costs of head_and_costs (App. B.3); removals int32 [P, B]."""
        if not hasattr(self, "_blocks_dev"):
            self._blocks_dev = torch.tensor(self.prune, dtype=torch.int32,
                                            device=self.cost.device)
        return dora_step_rewards(self.cost, removals, self._blocks_dev, self.depth,
                                 self.n_tokens - 1, a, reward, ret=ret, stream=stream)

    def head_and_costs(self, x, cu, norm_w, norm_b, eps, w_head, b_head, lc1=False, tau=3.0,
                       stream=None):
        """Logits of every sequence (classes padded to a multiple of 32) and
        each one's fidelity cost against its image's Native logits (0 for the
        Native rows themselves; the rollout's row is the full prefix)."""
        n = cu.numel() - 1
        logits = self.logits[:n]
        head = dora_classifier_head_lc1 if lc1 else dora_classifier_head
        self.head_ws = head(x, cu, norm_w, norm_b, eps, w_head, b_head, logits, self.head_ws,
                            stream=stream)
        native = self.logits[self.b:2 * self.b]
        dora_kd_cost(native, logits, self.cost[:n], self.classes, shadow_image=self.image_of[:n],
                     tau=tau, status=self.status, stream=stream)
        return logits, self.cost[:n]


__all__ = ["ShadowRollout"]
