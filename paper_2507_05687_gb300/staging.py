"""Overlapped host-to-device staging of training batches (host logic).

A training loop that feeds each GRPO step from pinned host memory pays the
copy of the step's batch (H alone is 268 MB at the 8B batch) on the step's
critical path.  BatchStager copies the next batch on a copy stream while the
current step computes: submit() enqueues the copies of one batch into a
device slot (slots are reused round robin, each only after the step that read
it has finished), get() hands the oldest submitted batch to the compute
stream, which waits for its copies first.  The copies run on the copy
engines, so the step's kernels keep every SM.  Nothing here computes: the
steps themselves are the library's calls on the returned device tensors.
"""
from __future__ import annotations

from collections import deque
from typing import Deque, List, Optional, Sequence

import torch


class BatchStager:
    """Round-robin device slots for batches of pinned host tensors.

    slots: device copies of a batch that may exist at once (2: the batch being
    computed and the next one in flight)."""

    def __init__(self, device: torch.device, slots: int = 2):
        if slots < 2:
            raise ValueError("slots >= 2 (one computing, one in flight)")
        self.device = torch.device(device)
        self.stream = torch.cuda.Stream(self.device)
        self._slots: List[Optional[List[torch.Tensor]]] = [None] * slots
        self._released: List[Optional[torch.cuda.Event]] = [None] * slots
        self._pending: Deque[tuple] = deque()  # (slot, copies-done event)
        self._next = 0
        self._current: Optional[int] = None  # the slot get() handed out and release() has not marked yet

    def submit(self, host_tensors: Sequence[torch.Tensor]) -> None:
        """Start copying one batch (pinned host tensors, any dtypes and shapes)
        into the next slot.  Raises if every slot is still taken (submitted
        and not yet handed out by get())."""
        if len(self._pending) >= len(self._slots):
            raise RuntimeError("every slot holds a batch not yet taken by get()")
        if any(h.device.type != "cpu" for h in host_tensors):
            raise ValueError("submit() takes host tensors")
        slot = self._next
        if slot == self._current:
            raise RuntimeError("the next slot's batch is still in use: release() it first")
        self._next = (self._next + 1) % len(self._slots)
        bufs = self._slots[slot]
        if bufs is None or len(bufs) != len(host_tensors) or any(
                b.shape != h.shape or b.dtype != h.dtype for b, h in zip(bufs, host_tensors)):
            bufs = [torch.empty(h.shape, dtype=h.dtype, device=self.device) for h in host_tensors]
            self._slots[slot] = bufs
        with torch.cuda.stream(self.stream):
            if self._released[slot] is not None:  # the step that last read this slot is done with it
                self.stream.wait_event(self._released[slot])
            for b, h in zip(bufs, host_tensors):
                b.copy_(h, non_blocking=True)
            done = torch.cuda.Event()
            done.record(self.stream)
        self._pending.append((slot, done))

    def get(self) -> List[torch.Tensor]:
        """The oldest submitted batch as device tensors; the current stream of
        the device waits for its copies.  Call release() once the work that
        reads them has been enqueued (before the slot's next submit)."""
        if not self._pending:
            raise RuntimeError("no batch submitted")
        if self._current is not None:
            raise RuntimeError("release() the previous batch first")
        slot, done = self._pending.popleft()
        torch.cuda.current_stream(self.device).wait_event(done)
        self._current = slot
        return self._slots[slot]

    def release(self) -> None:
        """Mark the batch last returned by get() as read by everything enqueued
        so far on the current stream: its slot is refilled only after that."""
        if self._current is None:
            raise RuntimeError("no batch handed out")
        ev = torch.cuda.Event()
        ev.record(torch.cuda.current_stream(self.device))
        self._released[self._current] = ev
        self._current = None
