"""Host-side pieces of the chain driver that need no GPU: the row copy into a hop's slot of the
chain buffer, and starting a chain afresh."""
import torch

from paper_2609_32046_gb300 import Chain, _copy_rows


def test_copy_rows_fills_only_the_slot():
    g = torch.Generator().manual_seed(3)
    buf = torch.zeros(2, 3, 40, 16, dtype=torch.bfloat16)
    src = torch.randn(2, 3, 11, 16, generator=g).to(torch.bfloat16)
    _copy_rows(buf[:, :, 7:18], src)
    assert torch.equal(buf[:, :, 7:18].view(torch.int16), src.view(torch.int16))   # bit-exact
    assert buf[:, :, :7].abs().sum() == 0 and buf[:, :, 18:].abs().sum() == 0


def test_copy_rows_falls_back_for_strided_rows():
    g = torch.Generator().manual_seed(4)
    buf = torch.zeros(2, 3, 20, 12, dtype=torch.bfloat16)
    src = torch.randn(2, 3, 12, 16, generator=g).to(torch.bfloat16).transpose(2, 3)   # rows not contiguous
    assert src.stride(-1) != 1
    _copy_rows(buf[:, :, 2:18], src)
    assert torch.equal(buf[:, :, 2:18], src)
    assert buf[:, :, :2].abs().sum() == 0 and buf[:, :, 18:].abs().sum() == 0


def test_chain_reset_starts_without_a_message():
    ch = Chain.__new__(Chain)           # the buffers are not needed to check the bookkeeping
    ch.cur, ch.T_old, ch.capacity = 1, 1234, 4096
    ch.reset()
    assert ch.cur == 0 and ch.T_old == 0
