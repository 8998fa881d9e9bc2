"""Search loops over the C ABI (host orchestration only; every step runs in the library).

* best-of-N exploration and selection (Algorithm 1), with an optional full-compute
  commit of the winner (tau = 0, the "commit" branch);
* beam-style rescoring: every ``every`` steps keep the top ``keep`` candidates and refill
  each with ``children`` perturbed copies (cs_beam_refill);
* pruned search (Sec. abl-stack): prune to the top ``keep`` at ``prune_step`` and continue;
* the static every-k-th-step schedule (Sec. 3.1, Properties), applied as a forced mask.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as B


def time_grid(T: int) -> np.ndarray:
    """t_k = 1 - (k-1)/T, k = 1..T+1."""
    return 1.0 - np.arange(T + 1, dtype=np.float64) / T


def static_schedule(k: int, T: int, K_w: int, K_c: int, every: int) -> bool:
    """Uniform schedule: warmup/cooldown compute; between them every ``every``-th step
    counted from the end of the warmup."""
    if k <= K_w or k > T - K_c:
        return True
    return (k - K_w) % every == 0


class Search:
    """Device state of up to ``max_n`` candidates plus the buffers a search needs."""

    def __init__(self, model: B.Model, max_n: int, target=None, device="cuda"):
        self.model = model
        self.D = model.mcfg.D
        self.max_n = max_n
        self.bufs = [B.new_state(max_n, self.D, device), B.new_state(max_n, self.D, device)]
        self.cur = 0
        self.n = max_n
        self.skip = torch.zeros(max_n, dtype=torch.uint8, device=device)
        self.scores = torch.zeros(max_n, device=device)
        self.top = torch.zeros(max_n, dtype=torch.int32, device=device)
        self.force = torch.zeros(max_n, dtype=torch.uint8, device=device)
        self.target = target
        self.ids = np.arange(max_n)        # original candidate index of each slot

    @property
    def st(self):
        full = self.bufs[self.cur]
        return {k: v[:self.n] for k, v in full.items()}

    def reset(self, x1):
        """Fresh search from latents x1 [N, D] (device tensor)."""
        self.cur = 0
        self.n = x1.shape[0]
        st = self.bufs[0]
        st["x"][:self.n].copy_(x1)
        st["has_ref"].zero_()
        st["accum"].zero_()
        self.ids = np.arange(self.n)

    def step(self, k, T, tau, K_w, K_c, score=False, force=None, schedule_every=0) -> int:
        t = time_grid(T)
        f = None
        if force is not None:
            self.force[:self.n].copy_(force)
            f = self.force[:self.n]
        elif schedule_every:
            self.force[:self.n].fill_(1 if static_schedule(k, T, K_w, K_c, schedule_every) else 0)
            f = self.force[:self.n]
        return self.model.search_step(self.st, k, T, float(t[k - 1]), float(t[k]), tau, K_w, K_c,
                                      self.skip[:self.n], force=f,
                                      target=self.target if score else None,
                                      scores=self.scores[:self.n] if score else None)

    def select(self, keep: int):
        """Indices (slots) of the ``keep`` best current scores, descending (device)."""
        B.select_topk(self.scores[:self.n], keep, self.top)
        return self.top[:keep]

    def refill(self, survivors, children: int, sigma: float, noise=None):
        """Keep ``survivors`` (device int32 slots) and give each ``children`` perturbed
        copies; the new population has len(survivors) * (1 + children) candidates."""
        keep = survivors.numel()
        src = self.st
        dst_full = self.bufs[1 - self.cur]
        B.beam_refill(src, dst_full, survivors, children, sigma, noise)
        surv = survivors.cpu().numpy()
        self.ids = np.repeat(self.ids[surv], children + 1)
        self.cur = 1 - self.cur
        self.n = keep * (children + 1)

    # ------------------------------------------------------------ searches --
    def best_of_n(self, x1, T, tau, K_w, K_c, schedule_every=0, forces=None):
        """Algorithm 1 exploration.  Returns (winner's candidate index, scores, skip masks)."""
        self.reset(x1)
        masks = []
        for k in range(1, T + 1):
            self.step(k, T, tau, K_w, K_c, score=(k == T), schedule_every=schedule_every,
                      force=None if forces is None else forces[k - 1])
            masks.append(self.skip[:self.n].cpu().numpy().astype(bool))
        best = int(self.select(1)[0])
        return int(self.ids[best]), self.scores[:self.n].cpu().numpy(), np.array(masks)

    def beam(self, x1, T, tau, K_w, K_c, every, keep, children, sigma, noise_rounds):
        """Beam-style search; noise_rounds[r] is the device noise [keep*children, D] of refill r."""
        self.reset(x1)
        r = 0
        for k in range(1, T + 1):
            rescore = (k % every == 0 and k < T) or k == T
            self.step(k, T, tau, K_w, K_c, score=rescore)
            if k % every == 0 and k < T:
                self.refill(self.select(keep).clone(), children, sigma, noise_rounds[r])
                r += 1
        best = int(self.select(1)[0])
        return best, self.scores[:self.n].cpu().numpy()

    def pruned(self, x1, T, tau, K_w, K_c, prune_step, keep):
        """Sec. abl-stack: prune to the top ``keep`` at ``prune_step``.  Returns the winner's
        original candidate index and the survivors' final scores and indices."""
        self.reset(x1)
        for k in range(1, T + 1):
            prune = k == prune_step
            self.step(k, T, tau, K_w, K_c, score=(prune or k == T))
            if prune:
                self.refill(self.select(keep).clone(), 0, 0.0, None)
        best = int(self.select(1)[0])
        return int(self.ids[best]), self.scores[:self.n].cpu().numpy(), self.ids.copy()

    def commit(self, x1_winner, T, K_w, K_c):
        """Algorithm 1 commit branch: the winner's seed again at full compute (tau = 0)."""
        self.reset(x1_winner)
        for k in range(1, T + 1):
            self.step(k, T, 0.0, K_w, K_c)
        return self.st["x"][0].clone()
