"""GPU: the L2-flush writer (Section 2.1, Section 4.2 region entry) writes
exactly the bytes it is given, every one of them, and nothing past them; each
call writes a different value, so no store can be elided as redundant."""
import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


def _flush_after_fill(fill, nbytes, pad=4096):
    buf = torch.full((nbytes + pad,), fill, dtype=torch.uint8, device="cuda")
    krex.krex_flush_l2(buf, nbytes)
    torch.cuda.synchronize()
    return buf.cpu().numpy()


# empty, tail only, whole words, words plus a tail, several grid strides
@pytest.mark.parametrize("nbytes", [0, 1, 15, 16, 17, 8192 + 5, 3 * (1 << 20) + 16 * 7 + 9, (160 << 20) + 3])
def test_flush_writes_exactly_its_bytes(nbytes):
    n16, ntail = divmod(nbytes, 16)
    seen = []
    for fill in (0xA5, 0x5A):
        h = _flush_after_fill(fill, nbytes)
        assert np.all(h[nbytes:] == fill)                 # nothing past the end
        words = h[:n16 * 16].reshape(-1, 16)
        if n16:
            assert np.all(words == words[0])              # every word written alike
            assert not np.all(words[0] == fill)
        tail = h[n16 * 16:nbytes]
        assert np.all(tail == tail[:1])
        seen.append((words[:1].tobytes(), tail.tobytes()))
    if nbytes:
        assert seen[0] != seen[1]                         # a fresh value on every call
    if ntail:
        # an unwritten tail would hold each call's fill byte
        assert not (seen[0][1] == bytes([0xA5]) * ntail and seen[1][1] == bytes([0x5A]) * ntail)


def test_flush_rejects_unaligned_scratch_without_writing():
    buf = torch.full((4096,), 0x33, dtype=torch.uint8, device="cuda")
    with pytest.raises(krex.KrexError, match="UNSUPPORTED"):
        krex.krex_flush_l2(buf.data_ptr() + 4, 1024)
    with pytest.raises(krex.KrexError, match="INVALID"):
        krex.krex_flush_l2(0, 1024)
    torch.cuda.synchronize()
    assert torch.all(buf == 0x33).item()
