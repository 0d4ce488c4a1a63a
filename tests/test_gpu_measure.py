"""voxzip_stream_read, the measurement helper bench.py times its ceilings with: it reads a device
buffer with 16-byte loads and stores only a checksum that no input here produces, so its sink stays
zero and the status word clean; a captured loop of it replays (needs a GB300)."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_08569_gb300 import build
    build.build_library()


@pytest.mark.parametrize("nbytes", [16, 4096 + 16, 3 << 20, 257 << 20])
def test_stream_read_reads_and_leaves_the_sink(nbytes):
    from paper_2608_08569_gb300 import voxzip_get_status, voxzip_stream_read
    buf = torch.zeros(nbytes // 4, dtype=torch.int32, device="cuda")
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    voxzip_get_status()
    voxzip_stream_read(buf, nbytes, sink)
    torch.cuda.synchronize()
    assert voxzip_get_status() == 0
    assert int(sink.item()) == 0


def test_stream_read_in_a_graph_loop():
    from paper_2608_08569_gb300 import voxzip_stream_read
    buf = torch.zeros(1 << 20, dtype=torch.int32, device="cuda")
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        voxzip_stream_read(buf, 4 << 20, sink)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for _ in range(8):
            voxzip_stream_read(buf, 4 << 20, sink)
    g.replay()
    torch.cuda.synchronize()
    assert int(sink.item()) == 0


def test_stream_read_rejects_sizes_beyond_the_buffer():
    from paper_2608_08569_gb300 import voxzip_stream_read
    buf = torch.zeros(64, dtype=torch.int32, device="cuda")
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(ValueError):
        voxzip_stream_read(buf, 1024, sink)
