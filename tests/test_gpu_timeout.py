"""The decoder's own bounded waits.

A decoder created with a wait limit of one SM cycle gives up on the first barrier wait that
does not complete at once (a weight copy or an MMA still in flight): the CTA raises its abort
flag, issues nothing more, drains what it had started (with a bound of its own, independent of
the caller's limit) and exits.  aecct_synchronize then reports AECCT_ERR_TIMEOUT.  The context
stays usable: a decoder with the default limit, created afterwards, decodes bit for bit as the
oracle does.  No wait is made to hang and nothing faults: every wait here is bounded, and the
short limit only makes the bound small.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

torch = pytest.importorskip("torch")


@pytest.mark.gpu
@pytest.mark.parametrize("key,B,cluster_ctas", [
    ("polar64_32", 4096, 0),    # d = 64, one CTA per word
    ("bch63_36", 1024, 0),      # d = 128 weight schedule (region U, operand-tile halves)
    ("ldpc384_192", 64, 0),     # d = 128 over a 5-CTA cluster (peers wait on each other)
])
def test_short_wait_limit_reports_timeout_and_context_survives(key, B, cluster_ctas):
    w = I.workload(key)
    model = I.workload_model(key)
    y = I.channel_batch(w.code, B, w.ebn0_db[0], seed=61).y
    yt = torch.from_numpy(y).cuda()
    short = A.Decoder(model, cluster_ctas=cluster_ctas, wait_limit_cycles=1)
    short.decode(yt)
    torch.cuda.synchronize()
    assert short.synchronize() == A.AECCT_ERR_TIMEOUT
    assert "wait" in A.last_error()
    # the status was reported once; the handle itself stays valid
    assert short.synchronize() == A.AECCT_OK
    short.close()
    # a normal decoder on the same context decodes exactly
    dec = A.Decoder(model, cluster_ctas=cluster_ctas)
    bits, syn, logits = dec.decode(yt[:8])
    torch.cuda.synchronize()
    assert dec.synchronize() == A.AECCT_OK
    ref = O.decode(model, y[:8])
    assert (logits.cpu().numpy().view(np.int32) == ref["logits"].view(np.int32)).all()
    assert (bits.cpu().numpy() == ref["bits"]).all() and (syn.cpu().numpy() == ref["syndrome"]).all()
    dec.close()
