"""spire_stream_read: the one-launch read floor the benchmark reports beside
calls that move tens of MB.  It computes nothing, so the test checks that it
runs to completion on ragged sizes (a final partial chunk, fewer chunks than
SMs) and leaves the buffer it reads untouched."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("nbytes", [16, 4096, 16384 * 3 + 48, 138 << 20])
def test_stream_read_runs_and_reads_only(nbytes):
    import paper_2504_06419_gb300 as spire
    buf = torch.arange((nbytes + 3) // 4, dtype=torch.int32, device="cuda")
    before = buf.clone()
    assert spire.spire_stream_read(buf, nbytes) == 0
    torch.cuda.synchronize()
    assert torch.equal(buf, before)
