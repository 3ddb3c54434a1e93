"""The training-time AAP weight quantiser (Sec. 4.1, eq. Ternary) on the GPU (aecct_aap_ternarize)
against the oracle's oracle_ternary, bit for bit: the 2-bit codes, the scale gamma * delta and the
forward weights scale * Ternary(W).  Then a model whose fp32 weights are quantised on the GPU
decodes exactly as the oracle decodes the same weights quantised by the oracle."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2410_05911_gb300 import aecct as A
from paper_2410_05911_gb300 import inputs as I

torch = pytest.importorskip("torch")


def _unpack(codes: np.ndarray) -> np.ndarray:
    c = codes.astype(np.uint8)
    fields = np.stack([(c >> (2 * i)) & 3 for i in range(4)], 1).reshape(-1)
    assert not (fields == 2).any()
    return np.where(fields == 1, 1, np.where(fields == 3, -1, 0)).astype(np.int8)


def _tensors(seed):
    rng = np.random.default_rng(seed)
    out = [
        (rng.standard_normal((128, 128)) / np.sqrt(128)).astype(np.float32),  # d x d
        (rng.standard_normal((512, 128)) / np.sqrt(128)).astype(np.float32),  # F x d
        (rng.standard_normal((32, 128)) / np.sqrt(128)).astype(np.float32),   # d x F at d = 32
        np.array([0.5, -0.25, 0.25, -0.5], np.float32),                       # the smallest tensor
        np.round(rng.standard_normal((64, 64)) * 4) / 4,                      # many ties in |W|
        np.zeros((16, 16), np.float32),                                        # gamma = 0
        np.where(rng.random((32, 32)) < 0.5, -0.0, 0.75).astype(np.float32),   # signed zeros
        (rng.standard_normal((1000, 4)) * 1e-20).astype(np.float32),           # tiny values
    ]
    return [np.ascontiguousarray(t, np.float32) for t in out]


@pytest.mark.gpu
@pytest.mark.parametrize("delta,eps", [(1.0, 1e-8), (2.0, 1e-8), (1.555, 1e-5), (0.7, 1e-30)])
def test_aap_ternarize_matches_oracle(delta, eps):
    ts = _tensors(int(delta * 1000))
    deltas = np.full(len(ts), delta, np.float32)
    deltas[1] = 1.25  # a different delta for one tensor
    codes, scale, wq = A.aap_ternarize([torch.from_numpy(t).cuda() for t in ts], deltas, eps, want_weights=True)
    torch.cuda.synchronize()
    sc = scale.cpu().numpy()
    for j, t in enumerate(ts):
        ref_t, ref_sc = O.ternary(t, delta=float(deltas[j]), eps=eps)
        got_t = _unpack(codes[j].cpu().numpy())
        assert (got_t == ref_t.reshape(-1)).all(), f"tensor {j}: {(got_t != ref_t.reshape(-1)).sum()} codes differ"
        assert sc[j].view(np.int32) == np.float32(ref_sc).view(np.int32), f"tensor {j}: scale {sc[j]} vs {ref_sc}"
        want_w = (np.float32(ref_sc) * ref_t.astype(np.float32)).reshape(-1)
        assert (wq[j].cpu().numpy().reshape(-1).view(np.int32) == want_w.view(np.int32)).all()


@pytest.mark.gpu
def test_aap_ternarize_more_tensors_than_one_launch():
    rng = np.random.default_rng(5)
    ts = [(rng.standard_normal(4 * (1 + j % 7)) + j).astype(np.float32) for j in range(150)]
    codes, scale, _ = A.aap_ternarize([torch.from_numpy(t).cuda() for t in ts], np.ones(150, np.float32), 1e-8)
    torch.cuda.synchronize()
    for j, t in enumerate(ts):
        ref_t, ref_sc = O.ternary(t, delta=1.0, eps=1e-8)
        assert (_unpack(codes[j].cpu().numpy()) == ref_t).all() and scale[j].item() == ref_sc


@pytest.mark.gpu
def test_model_quantised_on_gpu_decodes_like_the_oracle():
    # fp32 weights quantised by eq. Ternary on the GPU feed aecct_create; the oracle decodes the
    # same fp32 weights quantised by its own oracle_ternary
    code = I.make_code("bch31_16")
    base = I.random_model(code, 32, 2, seed=3, full_precision=True)
    deltas = np.array([[2.0, 1.9, 2.1, 1.8, 2.2, 2.0]] * base.n_layers, np.float32)
    flat = [torch.from_numpy(np.ascontiguousarray(w)).cuda() for wl in base.w_full for w in wl]
    codes, scale, _ = A.aap_ternarize(flat, deltas.reshape(-1), 1e-8)
    torch.cuda.synchronize()
    gpu_model = I.random_model(code, 32, 2, seed=3)  # the same biases, LN, embedding, head
    ora_model = I.random_model(code, 32, 2, seed=3)
    sc = scale.cpu().numpy().reshape(base.n_layers, 6)
    for l in range(base.n_layers):
        for g in range(6):
            w = base.w_full[l][g]
            gpu_model.w_tern[l][g] = _unpack(codes[6 * l + g].cpu().numpy()).reshape(w.shape)
            t, s = O.ternary(w, delta=float(deltas[l, g]), eps=1e-8)
            ora_model.w_tern[l][g] = t.reshape(w.shape)
            ora_model.w_scale[l, g] = s
    gpu_model.w_scale = sc.astype(np.float32)
    assert all((a == b).all() for la, lb in zip(gpu_model.w_tern, ora_model.w_tern) for a, b in zip(la, lb))
    y = I.channel_batch(code, 40, 4.0, seed=9).y
    dec = A.Decoder(gpu_model)
    bits, syn, logits = dec.decode(torch.from_numpy(y).cuda())
    torch.cuda.synchronize()
    assert dec.synchronize() == A.AECCT_OK
    ref = O.decode(ora_model, y)
    assert (logits.cpu().numpy().view(np.int32) == ref["logits"].view(np.int32)).all()
    assert (bits.cpu().numpy() == ref["bits"]).all()
    dec.close()
