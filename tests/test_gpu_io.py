"""Staging copies (cmc_stage_copies) on the GPU: pinned host <-> device and
device <-> device byte ranges, copied exactly, in both ordering modes, and
their place in stream order (a launch completes after the kernel before it,
so a copy enqueued after it sees that kernel's writes)."""

import numpy as np
import pytest
import torch

import paper_2609_25537_gb300 as cmc

pytestmark = pytest.mark.gpu


def _bytes(n, seed):
    return torch.from_numpy(np.random.default_rng(seed).integers(0, 256, n, dtype=np.uint8))


@pytest.mark.parametrize("wait_first", [False, True])
def test_host_device_round_trip(cuda_device, wait_first):
    sizes = [16, 4096 + 48, 3 << 20, 1 << 16]
    h_in = [_bytes(n, i).pin_memory() for i, n in enumerate(sizes)]
    d = [torch.empty(n, dtype=torch.uint8, device=cuda_device) for n in sizes]
    cmc.stage_copies(list(zip(h_in, d)), wait_first=wait_first)
    h_out = [torch.empty(n, dtype=torch.uint8).pin_memory() for n in sizes]
    cmc.stage_copies(list(zip(d, h_out)), wait_first=True)
    torch.cuda.synchronize()
    for a, dev_t, b in zip(h_in, d, h_out):
        assert torch.equal(dev_t.cpu(), a)
        assert torch.equal(b, a)


def test_device_to_device_and_empty(cuda_device):
    src = _bytes(1 << 20, 7).to(cuda_device)
    dst = torch.zeros_like(src)
    empty = torch.empty(0, dtype=torch.uint8, device=cuda_device)
    cmc.stage_copies([(src, dst), (empty, empty)])
    cmc.stage_copies([])
    torch.cuda.synchronize()
    assert torch.equal(src, dst)


def test_stream_order_with_a_writing_kernel(cuda_device):
    """A buffer written by a kernel, then copied to the host with
    wait_first=True, arrives as written; a no-wait copy enqueued after that
    one completes after it, so the host sees both."""
    s = torch.cuda.current_stream(cuda_device)
    a = torch.empty(1 << 20, dtype=torch.uint8, device=cuda_device)
    b = _bytes(1 << 16, 3).pin_memory()
    b_dev = torch.empty(1 << 16, dtype=torch.uint8, device=cuda_device)
    h = torch.empty(1 << 20, dtype=torch.uint8).pin_memory()
    for v in (5, 9, 13):
        a.fill_(v)                                              # the writing kernel
        cmc.stage_copies([(a, h)], wait_first=True)             # waits for it
        cmc.stage_copies([(b, b_dev)], wait_first=False)        # independent of it
        s.synchronize()
        assert int(h.min()) == v and int(h.max()) == v
        assert torch.equal(b_dev.cpu(), b)


def test_rejects_unpinned_host_memory(cuda_device):
    with pytest.raises(ValueError, match="pinned"):
        cmc.stage_copies([(torch.zeros(64, dtype=torch.uint8),
                           torch.zeros(64, dtype=torch.uint8, device=cuda_device))])
