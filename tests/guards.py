"""Guard regions around device outputs (test infrastructure; a stand-in for a
memory checker): every buffer allocated here sits between two 4 KB canaries of known
bytes, and after each GPU test the canaries must be untouched, so a kernel that
writes past either end of an output or workspace fails the test that ran it."""
from __future__ import annotations

import math

import torch

PAD = 4096  # bytes on each side; keeps the buffer 256-byte aligned like a fresh allocation
LO, HI = 0xA5, 0x5A

_live: list[tuple[torch.Tensor, int, str]] = []


def empty(shape, dtype, fill=None, what: str = "") -> torch.Tensor:
    shape = tuple(shape)
    nbytes = math.prod(shape) * torch.empty((), dtype=dtype).element_size()
    raw = torch.empty(nbytes + 2 * PAD, dtype=torch.uint8, device="cuda")
    raw[:PAD].fill_(LO)
    raw[PAD + nbytes:].fill_(HI)
    t = raw[PAD:PAD + nbytes].view(dtype).view(shape)
    if fill is not None:
        t.fill_(fill)
    _live.append((raw, nbytes, what or f"{dtype} {shape}"))
    return t


def like(t: torch.Tensor, fill=None) -> torch.Tensor:
    return empty(t.shape, t.dtype, fill)


def zeros(shape, dtype) -> torch.Tensor:
    return empty(shape, dtype, 0)


def check_and_clear():
    """Every canary written since the last call must still hold its bytes."""
    if not _live:
        return
    torch.cuda.synchronize()
    bad = []
    for raw, nbytes, what in _live:
        if not (bool((raw[:PAD] == LO).all()) and bool((raw[PAD + nbytes:] == HI).all())):
            bad.append(what)
    _live.clear()
    assert not bad, f"guard bytes overwritten around: {bad}"
