"""Host-side layout logic of the Python binding (CPU only)."""
import torch

from paper_2609_29029_gb300.pipeline import interleave_gate_up


def test_gate_up_rows_interleave_in_groups_of_sixteen():
    """The SwiGLU epilogue reads 16 gate rows and then the 16 matching up rows of every 32-row
    group: row 32 k + j is gate row 16 k + j and row 32 k + 16 + j is up row 16 k + j."""
    F, d = 64, 8
    wg = torch.arange(F * d, dtype=torch.float32).view(F, d)
    wu = -wg - 1
    w = interleave_gate_up(wg, wu)
    assert w.shape == (2 * F, d) and w.is_contiguous()
    for k in range(F // 16):
        assert torch.equal(w[32 * k:32 * k + 16], wg[16 * k:16 * k + 16])
        assert torch.equal(w[32 * k + 16:32 * k + 32], wu[16 * k:16 * k + 16])
