"""The measurement probe of the bench's practical ceiling reads exactly the
pieces it is given (GPU)."""
import numpy as np
import pytest
import torch

from gpu_util import DEV, to_dev
from paper_2606_03026_gb300 import spikeproj as sp

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("piece", [512, 1024, 1536])
@pytest.mark.parametrize("count", [0, 1, 4863, 4864, 4865, 77821])
def test_probe_reads_the_listed_pieces(count, piece):
    """The XOR of every word the probe reads equals the XOR of the listed
    pieces (a piece listed twice cancels, as it does on the host)."""
    rng = np.random.default_rng(count)
    nbytes = 1 << 22
    buf = rng.integers(0, 1 << 32, size=nbytes // 4, dtype=np.uint32)
    offs = rng.integers(0, (nbytes - piece) // 16, size=count).astype(np.uint32)
    want = np.uint32(0)
    words = buf.view(np.uint32)
    for o in offs:
        want ^= np.bitwise_xor.reduce(words[o * 4: o * 4 + piece // 4])
    sink = torch.zeros(1, dtype=torch.int32, device=DEV)
    dbuf = to_dev(buf)
    doffs = to_dev(offs) if count else torch.zeros(1, dtype=torch.int32, device=DEV)
    sp.spike_proj_probe_gather(dbuf, doffs, count, sink, piece_bytes=piece)
    torch.cuda.synchronize()
    assert np.uint32(sink.cpu().numpy().view(np.uint32)[0]) == want


def test_probe_argument_errors():
    sink = torch.zeros(1, dtype=torch.int32, device=DEV)
    buf = torch.zeros(1024, dtype=torch.uint8, device=DEV)
    with pytest.raises(sp.SpikeProjError) as e:
        sp.spike_proj_probe_gather(buf, None, 3, sink)
    assert e.value.status == sp.SP_EINVAL
    with pytest.raises(sp.SpikeProjError) as e:
        sp.spike_proj_probe_gather(buf[1:], None, 0, sink)
    assert e.value.status == sp.SP_EALIGN
