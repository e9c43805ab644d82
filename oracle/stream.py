"""Rolling-window history update (Sec. 3.1; Algorithm 1, KV update with the
stop-gradient head prediction). Test infrastructure.

After each pass the head state (window position 1, fine scale) is emitted and
its K/V join the history cache; the sink never changes. The cache has a fixed
capacity: while it is not full a new frame takes the next free slot; once it
is full the new frame replaces the oldest one in place. Attention reads the
history in slot order (0 .. count-1); since softmax attention is invariant
to the order of its keys, slot order and age order give the same result up
to rounding, and slot order lets the cache be updated without moving data.
The oracle keeps no pooled copies: every pass recomputes its context from
the fine frames, which independently checks any incremental pyramid.
"""
from __future__ import annotations

import numpy as np


class History:
    def __init__(self, k_hist: np.ndarray, v_hist: np.ndarray, capacity: int):
        """k_hist/v_hist [B, n0, G, H, D]: the initial frames, oldest first."""
        B, n0, G, H, D = k_hist.shape
        if n0 > capacity:
            raise ValueError("more initial frames than capacity")
        self.capacity = capacity
        self.k = np.zeros((B, capacity, G, H, D), dtype=np.float64)
        self.v = np.zeros((B, capacity, G, H, D), dtype=np.float64)
        self.k[:, :n0] = k_hist
        self.v[:, :n0] = v_hist
        self.count = n0
        self.oldest = 0  # slot of the oldest frame once the cache is full

    def frames(self):
        """(k, v) of the live frames in slot order, [B, count, G, H, D]."""
        return self.k[:, :self.count], self.v[:, :self.count]

    def append(self, k_head: np.ndarray, v_head: np.ndarray) -> int:
        """Insert the emitted head's fine K/V [B, G, H, D]; returns the slot used."""
        if self.count < self.capacity:
            slot = self.count
            self.count += 1
        else:
            slot = self.oldest
            self.oldest = (self.oldest + 1) % self.capacity
        self.k[:, slot] = k_head
        self.v[:, slot] = v_head
        return slot
