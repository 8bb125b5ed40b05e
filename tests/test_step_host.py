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


@pytest.mark.parametrize("n_chunks", [1, 2, 3, 4, 5, 9])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_chunk_plan_covers_the_step(n_chunks, seed):
    g = torch.Generator().manual_seed(seed)
    R = 11
    span = torch.randint(0, 17, (R,), generator=g, dtype=torch.int32)
    span[seed] = 0                       # empty spans are allowed
    cu = torch.zeros(R + 1, dtype=torch.int32)
    cu[1:] = torch.cumsum(span, 0)
    T = int(cu[-1])
    bounds, cu_chunk = step_mod.chunk_plan(cu, n_chunks)
    # contiguous, request-aligned, covering every request and position once
    assert bounds[0][0] == 0 and bounds[-1][1] == R
    for (a0, a1, s0, s1), (b0, b1, u0, u1) in zip(bounds, bounds[1:]):
        assert a1 == b0 and s1 == u0
    for r0, r1, t0, t1 in bounds:
        assert r0 <= r1 and t0 == int(cu[r0]) and t1 == int(cu[r1])
    assert len(bounds) <= n_chunks
    # each chunk's offsets are the step's, rebased to its first position
    off = 0
    for r0, r1, t0, t1 in bounds:
        part = cu_chunk[off:off + r1 - r0 + 1]
        assert torch.equal(part, cu[r0:r1 + 1] - cu[r0])
        off += r1 - r0 + 1
    assert off == cu_chunk.numel() <= 2 * R + 1
    # every chunk but the last ends at or before the end of its share of T
    shares = [T * c // n_chunks for c in range(1, n_chunks + 1)]
    for r0, r1, t0, t1 in bounds[:-1]:
        assert any(t1 <= sh for sh in shares[:-1])
