"""GPU parity of inference with a quantized layer (Algorithm 2's revert applied to tokens,
Sec. 3.2) through the C ABI: the packed code layout round-trips bit for bit, and
y = W^ x from kq_infer (online Hadamard transforms around a dequantizing product) is within
1e-5 (relative L2 per token) of the oracle's dense float64 W^ x."""
import numpy as np
import pytest
import torch

from oracle import kronq_oracle as ref

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()


def K():
    from paper_2607_07964_gb300 import kronq
    return kronq


def _layer(d_out, d_in, bits, group, seed):
    rng = np.random.default_rng(seed)
    ng = 1 if group == 0 else d_in // group
    codes = rng.integers(0, 2 ** bits, size=(d_out, d_in)).astype(np.uint8)
    scale = (rng.random((d_out, ng)) * 0.01 + 1e-3).astype(np.float32)
    zero = rng.integers(0, 2 ** bits, size=(d_out, ng)).astype(np.int32)
    s_x = np.exp(rng.standard_normal(d_in) * 0.5).astype(np.float32)
    s_g = np.exp(rng.standard_normal(d_out) * 0.5).astype(np.float32)
    su = np.where(rng.random(d_out) < 0.5, -1, 1).astype(np.int8)
    sv = np.where(rng.random(d_in) < 0.5, -1, 1).astype(np.int8)
    return codes, scale, zero, s_x, s_g, su, sv


def _dev(a, dt=None):
    t = torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    return t if dt is None else t.to(dt)


def _unpack(words, d_out, d_in, bits):
    pb = 4 if bits == 3 else bits
    cpw = 32 // pb
    w = words.view(np.uint32).reshape(d_out, d_in // cpw)
    out = np.zeros((d_out, d_in), np.uint8)
    for t in range(cpw):
        out[:, t::cpw] = (w >> np.uint32(t * pb)) & np.uint32((1 << pb) - 1)
    return out


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_pack_roundtrip(bits):
    codes = _layer(96, 384, bits, 128, bits)[0]
    packed = torch.empty(K().kq_packed_codes_bytes(96, 384, bits) // 4, dtype=torch.int32, device=DEV)
    K().kq_pack_codes(_dev(codes), bits, packed)
    torch.cuda.synchronize()
    assert np.array_equal(_unpack(packed.cpu().numpy(), 96, 384, bits), codes)


@pytest.mark.parametrize("d_out,d_in,bits,group,B", [
    (256, 256, 4, 0, 1), (512, 896, 3, 128, 3), (1024, 4096, 2, 128, 1), (448, 1024, 8, 128, 8),
    (224, 512, 4, 128, 5), (4096, 4096, 4, 128, 2), (14336, 512, 4, 128, 1), (512, 4096, 4, 128, 1),
    (2048, 1024, 3, 128, 1)])
def test_infer_matches_dense_reverted_layer(d_out, d_in, bits, group, B):
    codes, scale, zero, s_x, s_g, su, sv = _layer(d_out, d_in, bits, group, d_in + bits)
    x = np.random.default_rng(B).standard_normal((B, d_in)).astype(np.float32)
    want = ref.infer(codes, scale, zero, group, s_x, s_g, su, sv, x)
    packed = torch.empty(K().kq_packed_codes_bytes(d_out, d_in, bits) // 4, dtype=torch.int32, device=DEV)
    K().kq_pack_codes(_dev(codes), bits, packed)
    y = torch.full((B, d_out), float("nan"), device=DEV)
    ws = torch.empty(K().kq_infer_workspace(B, d_in, d_out), dtype=torch.uint8, device=DEV)
    info = torch.zeros(1, dtype=torch.int32, device=DEV)
    K().kq_infer(packed, _dev(scale), _dev(zero), d_out, d_in, bits, group, _dev(s_x), _dev(s_g),
                 _dev(su), _dev(sv), _dev(x), y, ws, info=info)
    torch.cuda.synchronize()
    assert K().kq_check(info)[0] == K().KQ_OK
    got = y.cpu().numpy().astype(np.float64)
    for b in range(B):
        assert np.linalg.norm(got[b] - want[b]) <= 1e-5 * np.linalg.norm(want[b]), b


@pytest.mark.parametrize("bits,B", [(4, 1), (2, 2)])
def test_infer_chain_on_one_stream(bits, B):
    """Three layers back to back on one stream, each reading the previous one's output: the
    launches overlap their predecessors (programmatic dependent launch), so this checks that
    x is read only after the layer before has written it. Each layer matches the oracle on
    the input it was given; a CUDA graph of the chain reproduces the direct run bit for bit."""
    d = 1024
    layers = [_layer(d, d, bits, 128, 100 + i) for i in range(3)]
    dev = []
    for codes, scale, zero, s_x, s_g, su, sv in layers:
        packed = torch.empty(K().kq_packed_codes_bytes(d, d, bits) // 4, dtype=torch.int32, device=DEV)
        K().kq_pack_codes(_dev(codes), bits, packed)
        dev.append((packed, _dev(scale), _dev(zero), _dev(s_x), _dev(s_g), _dev(su), _dev(sv)))
    x0 = _dev(np.random.default_rng(7).standard_normal((B, d)).astype(np.float32))
    ys = [torch.full((B, d), float("nan"), device=DEV) for _ in range(3)]
    wss = [torch.empty(K().kq_infer_workspace(B, d, d), dtype=torch.uint8, device=DEV) for _ in range(3)]

    def chain(s):
        inp = x0
        for i in range(3):
            p, sc, z, sx, sg, su, sv = dev[i]
            K().kq_infer(p, sc, z, d, d, bits, 128, sx, sg, su, sv, inp, ys[i], wss[i], stream=s)
            inp = ys[i]

    torch.cuda.synchronize()
    chain(torch.cuda.current_stream())
    torch.cuda.synchronize()
    got = [y.cpu().numpy().astype(np.float64) for y in ys]
    inp = x0.cpu().numpy()
    for i, (codes, scale, zero, s_x, s_g, su, sv) in enumerate(layers):
        want = ref.infer(codes, scale, zero, 128, s_x, s_g, su, sv, inp)
        for b in range(B):
            assert np.linalg.norm(got[i][b] - want[b]) <= 1e-5 * np.linalg.norm(want[b]), (i, b)
        inp = got[i].astype(np.float32)
    for y in ys:
        y.fill_(float("nan"))
    g = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    with torch.cuda.graph(g, stream=cap):
        chain(cap)
    g.replay()
    torch.cuda.synchronize()
    for i in range(3):
        assert np.array_equal(ys[i].cpu().numpy().astype(np.float64), got[i]), i
