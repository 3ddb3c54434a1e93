"""aecct_decode_host_noalloc (no paper counterpart): the host-buffer decode whose device staging
and status word come from the library's static scratch array instead of cudaMalloc.  It must
give exactly what aecct_decode_host gives, on two calls in a row (the status word is cleared
and the staging reused), and refuse a batch beyond the scratch with a clear error.  This file
is collected last and needs nothing from the other tests, so it also passes alone in a fresh
process."""
import numpy as np
import pytest

from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

pytest.importorskip("torch")


def _limit(n, m, syndrome=True, logits=True):
    r = lambda v: (v + 255) // 256 * 256  # noqa: E731
    best = 0
    for B in range(1, 1 << 16):
        end = 256 + r(4 * B * n) + r(B * n) + (r(B * m) if syndrome else 0) + (r(4 * B * n) if logits else 0)
        if end > (4 << 20):
            break
        best = B
    return best


@pytest.mark.gpu
@pytest.mark.parametrize("key,B", [("bch31_16", 300), ("polar64_32", 1000), ("bch63_36", 64)])
def test_noalloc_matches_host_entry_point_twice(key, B):
    w = I.workload(key)
    dec = A.Decoder(I.workload_model(key))
    y = I.channel_batch(w.code, B, w.ebn0_db[0], seed=31).y
    bits, syn, logits = dec.decode_host(y)
    for call in range(2):
        st, b2, s2, l2 = dec.decode_host_noalloc(y)
        assert st == A.AECCT_OK, (call, A.last_error())
        assert (b2 == bits).all() and (s2 == syn).all(), call
        assert (l2.view(np.int32) == logits.view(np.int32)).all(), call
    # optional outputs left out
    st, b3, s3, l3 = dec.decode_host_noalloc(y, want_syndrome=False, want_logits=False)
    assert st == A.AECCT_OK and s3 is None and l3 is None and (b3 == bits).all()
    dec.close()


@pytest.mark.gpu
def test_noalloc_limit_and_refusal():
    key = "polar64_32"
    w = I.workload(key)
    dec = A.Decoder(I.workload_model(key))
    n, m = w.code.n, w.code.n - w.code.k
    bmax = _limit(n, m)
    assert bmax == 6897  # the figure the header states
    y = I.channel_batch(w.code, bmax, w.ebn0_db[0], seed=5).y
    st, bits, _, _ = dec.decode_host_noalloc(y)
    assert st == A.AECCT_OK
    ref, _, _ = dec.decode_host(y)
    assert (bits == ref).all()
    yb = np.concatenate([y, y[:1]])
    st, _, _, _ = dec.decode_host_noalloc(yb)
    assert st == A.AECCT_ERR_INVALID_ARG
    assert "static scratch" in A.last_error()
    # without logits the same scratch takes more words
    assert _limit(n, m, logits=False) > bmax
    st, _, _, _ = dec.decode_host_noalloc(yb, want_logits=False)
    assert st == A.AECCT_OK
    dec.close()


@pytest.mark.gpu
def test_noalloc_reports_timeout_then_recovers():
    # the status word read back from the scratch: a handle whose waits give up after one cycle
    # reports AECCT_ERR_TIMEOUT; the word is cleared before the next call, which then succeeds
    key = "polar64_32"
    w = I.workload(key)
    model = I.workload_model(key)
    y = I.channel_batch(w.code, 2048, w.ebn0_db[0], seed=13).y
    short = A.Decoder(model, wait_limit_cycles=1)
    st, _, _, _ = short.decode_host_noalloc(y)
    assert st == A.AECCT_ERR_TIMEOUT
    short.close()
    dec = A.Decoder(model)
    bits, syn, logits = dec.decode_host(y)
    st, b2, s2, l2 = dec.decode_host_noalloc(y)
    assert st == A.AECCT_OK
    assert (b2 == bits).all() and (s2 == syn).all() and (l2.view(np.int32) == logits.view(np.int32)).all()
    dec.close()
