"""Host-side layout of the step's packed buffers (no GPU needed)."""
import pytest
import torch

step_mod = pytest.importorskip("paper_2609_36546_gb300.step")


def test_packed_views_alignment_and_mirror():
    g = torch.Generator().manual_seed(5)
    named = [("q", torch.randn(3, 4, 128, generator=g).to(torch.bfloat16)),
             ("cu", torch.tensor([0, 3, 7, 9], dtype=torch.int32)),
             ("empty", torch.zeros(0, dtype=torch.int32)),
             ("drv", torch.tensor([1, 0, 1], dtype=torch.uint8)),
             ("pt", torch.randint(0, 1000, (3, 17), generator=g, dtype=torch.int32)),
             ("f", torch.tensor([1.5, -2.0], dtype=torch.float32))]
    p = step_mod._Packed(named, "cpu")
    assert p.buf.dtype == torch.uint8 and p.buf.numel() % 256 == 0
    offs = {}
    for name, off, nb, dt, sh in p.layout:
        assert off % 256 == 0
        offs[name] = (off, nb)
    # slots in order, none overlapping
    spans = sorted(offs.values())
    for (o1, n1), (o2, _) in zip(spans, spans[1:]):
        assert o1 + n1 <= o2
    for name, t in named:
        v = p.views[name]
        assert v.dtype == t.dtype and v.shape == t.shape
        assert torch.equal(v.view(torch.uint8) if v.numel() else v, t.view(torch.uint8) if t.numel() else t)
    m = p.mirror("cpu")
    assert m.buf.data_ptr() != p.buf.data_ptr()
    assert torch.equal(m.buf, p.buf)
    for name, t in named:
        assert torch.equal(m.views[name].view(torch.uint8), t.view(torch.uint8))
    # a write through a view lands in the buffer that one copy moves
    m.views["cu"][1] = 42
    p.buf.copy_(m.buf)
    assert int(p.views["cu"][1]) == 42
