"""Dynamic batching (Sec. 5.2, Algorithm 2) as host logic over the graph walk.

Algorithm 2 adjusts the batch size B along the gradient of the inference
latency, halves it when the hardware or real-time constraints are violated,
doubles it for sparse inputs (bounded by memory) and halves it for inputs of
high computational intensity, until the latency stops changing.  The GPU work
(one timed sparoa_run_graph per evaluated B) is the caller's ``latency``
callback; the memory model M(B) is ``memory`` (sparoa_graph_workspace plus
the input, no device work).

Readings of the listing, where it is open:
  objective   the latency per image L(B) / B (minimising the batch latency
              itself would drive B to 1, against the stated aim of higher
              throughput); its gradient is taken in log B as the elasticity
              d log(L/B) / d log B from the last two evaluated sizes (a
              scale-free step: eta is in octaves per unit elasticity), and the
              first step, with one point only, probes upwards by eta octaves
  constraints "M(B) > M_max and L(B) > T" halves B when either is violated
              (the text: a batch that exceeds the memory is halved); the
              smallest violating B is remembered, and later steps go at most
              halfway from B to it (a bisection of the feasible boundary
              instead of a cycle of overshoot and halving)
  2B cap      "min(2B, M_max)" caps the doubled batch at the largest B whose
              M(B) fits M_max
  stopping    |L(B)/B - L(B_prev)/B_prev| <= eps * L(B_prev)/B_prev, an
              unchanged B, or max_iter iterations
Every evaluated point is recorded in the returned trace.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field


@dataclass
class BatchTrace:
    batch: int                       # B*
    steps: list = field(default_factory=list)   # (B, latency_s, per_image_s, mem_bytes, note)

    def as_dict(self):
        return {"batch": self.batch,
                "steps": [{"B": b, "latency_ms": round(l * 1e3, 4), "per_image_us": round(p * 1e6, 3),
                           "mem_mb": round(m / 2 ** 20, 1), "note": n} for b, l, p, m, n in self.steps]}


def memory_cap(memory, mem_max: float, b_min: int = 1, b_max: int = 512) -> int:
    """Largest B in [b_min, b_max] with memory(B) <= mem_max (memory is
    non-decreasing in B), or b_min when even that does not fit."""
    if memory(b_max) <= mem_max:
        return b_max
    lo, hi = b_min, b_max  # memory(lo) may not fit: then b_min is returned
    if memory(lo) > mem_max:
        return b_min
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if memory(mid) <= mem_max:
            lo = mid
        else:
            hi = mid
    return lo


def dynamic_batch(latency, memory, B0: int, *, sparsity: float, intensity: float,
                  s_thr: float = 0.5, c_thr: float | None = None, mem_max: float = math.inf,
                  t_realtime: float = math.inf, eta: float = 1.0, eps: float = 0.02,
                  b_min: int = 1, b_max: int = 512, max_iter: int = 32) -> BatchTrace:
    """Algorithm 2.  latency(B) -> seconds for one batch of B; memory(B) -> bytes.
    sparsity / intensity describe the input (Eq. 1 zero fraction, FLOPs per
    byte); c_thr None disables the intensity rule."""
    clamp = lambda b: max(b_min, min(b_max, int(b)))
    tr = BatchTrace(batch=clamp(B0))
    cap = memory_cap(memory, mem_max, b_min, b_max)

    def evaluate(b, note):
        L = latency(b)
        M = memory(b)
        tr.steps.append((b, L, L / b, M, note))
        return L, M

    B = clamp(B0)
    L, M = evaluate(B, "initial")
    bad = b_max + 1  # smallest batch seen to violate a constraint
    B_prev = L_prev = None
    for _ in range(max_iter):
        if B_prev is not None:
            l, lp = L / B, L_prev / B_prev
            if abs(l - lp) <= eps * lp or B == B_prev:
                break
        # gradient step on the per-image latency, in log B
        if B_prev is None or B == B_prev:
            g = -1.0
        else:
            g = (math.log(L / B) - math.log(L_prev / B_prev)) / (math.log(B) - math.log(B_prev))
        limit = (B + bad) // 2 if bad <= b_max else b_max
        B_new = clamp(min(round(B * 2.0 ** (-eta * g)), limit))
        if B_new == B:
            B_new = clamp(min(B + (1 if g < 0 else -1), limit))
        L_new, M_new = evaluate(B_new, "gradient step")
        # hardware and real-time constraints
        while (M_new > mem_max or L_new > t_realtime) and B_new > b_min:
            bad = min(bad, B_new)
            B_new = clamp(B_new // 2)
            L_new, M_new = evaluate(B_new, "halved: memory or deadline")
        # input-driven partitioning
        if sparsity > s_thr:
            B_adj = clamp(min(2 * B_new, cap, bad - 1))
            note = "doubled: sparse input"
        elif c_thr is not None and intensity > c_thr:
            B_adj = clamp(B_new // 2)
            note = "halved: intense input"
        else:
            B_adj, note = B_new, None
        if note is not None and B_adj != B_new:
            B_new = B_adj
            L_new, M_new = evaluate(B_new, note)
        B_prev, L_prev = B, L
        B, L, M = B_new, L_new, M_new
    tr.batch = B
    return tr
