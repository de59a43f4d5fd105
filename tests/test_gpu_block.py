"""GPU parity of the transformer-block path (Sec. 3.3 sensitivity, Sec. 5 W2 -> W3
allocation) through the C ABI:
  * per-sublayer raw and post-BiIP traces within 1e-5 of the oracle, and the allocation
    the oracle makes from its own scores;
  * every sublayer's codes, grids and zeros bit-identical to that sublayer run alone
    through LayerPipeline.run (shared H_X accumulation, concurrent lanes and the
    precomputed scales change nothing);
  * each sublayer's proxy loss within 1e-3 of the oracle's block pipeline.
"""
import numpy as np
import pytest
import torch

import kqsynth
from oracle import kronq_oracle as ref

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_07964_gb300 import build
    build.build()


def _dev_inputs(b):
    f = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(DEV).to(dt)  # noqa: E731
    return ({k: f(v, torch.bfloat16) for k, v in b["X"].items()}, {k: f(v, torch.bfloat16) for k, v in b["G"].items()},
            {k: f(v, torch.float32) for k, v in b["W"].items()}, {k: f(v, torch.int8) for k, v in b["sign_u"].items()},
            {k: f(v, torch.int8) for k, v in b["sign_v"].items()})


@pytest.fixture(scope="module")
def block():
    from paper_2607_07964_gb300.block import BlockQuantizer
    cfg = kqsynth.BLOCKS["tiny_block"]
    b = kqsynth.block_inputs(cfg)
    spec = kqsynth.block_spec(cfg)
    X, G, W, su, sv = _dev_inputs(b)
    q = BlockQuantizer(spec, cfg.group, cfg.block, cfg.damp, cfg.low_bits, cfg.high_bits, cfg.budget, lanes=3)
    bits, sc = q.run(X, G, W, su, sv)
    q.check()
    return cfg, b, spec, q, bits, sc, (X, G, W, su, sv)


def test_block_scores_and_allocation(block):
    cfg, b, spec, q, bits, sc, _ = block
    o = ref.block_scores(b["X"], b["G"], b["W"], spec)
    for name, _, _, _ in spec:
        g = sc[name]
        for i, key in enumerate(("trHX", "trHG", "s", "trHX_post", "trHG_post", "s_post")):
            assert abs(g[i] - o[name][key]) <= 1e-5 * abs(o[name][key]), (name, key)
    s_post = {n: o[n]["s_post"] for n, _, _, _ in spec}
    vals = sorted(s_post.values())
    assert min(b2 / a - 1 for a, b2 in zip(vals, vals[1:])) > 1e-4, "scores too close to rank robustly"
    params = {n: d_out * d_in for n, _, d_out, d_in in spec}
    want = ref.allocate_bits(s_post, params, cfg.low_bits, cfg.high_bits, cfg.budget)
    assert bits == want
    assert 2 in bits.values() and 3 in bits.values()


def test_block_sublayers_equal_single_layer_runs(block):
    from paper_2607_07964_gb300.pipeline import LayerPipeline
    cfg, _, spec, q, bits, _, (X, G, W, su, sv) = block
    for name, grp, d_out, d_in in spec:
        p = LayerPipeline(d_out, d_in, bits[name], cfg.group, cfg.block, cfg.damp, g_chunk_tokens=0)
        p.run(X[grp], G[name], W[name], su[name], sv[name])
        p.check()
        bp = q.pipes[name]
        assert torch.equal(p.codes, bp.codes), name
        assert torch.equal(p.scale, bp.scale), name
        assert torch.equal(p.zero, bp.zero), name


def test_block_lanes_do_not_change_results(block):
    from paper_2607_07964_gb300.block import BlockQuantizer
    cfg, _, spec, q, bits, _, (X, G, W, su, sv) = block
    q1 = BlockQuantizer(spec, cfg.group, cfg.block, cfg.damp, cfg.low_bits, cfg.high_bits, cfg.budget, lanes=1)
    bits1, _ = q1.run(X, G, W, su, sv)
    q1.check()
    assert bits1 == bits
    for name, _, _, _ in spec:
        assert torch.equal(q1.pipes[name].codes, q.pipes[name].codes), name


def test_block_proxy_loss_against_oracle(block):
    from paper_2607_07964_gb300 import kronq as K
    cfg, b, spec, q, bits, _, (X, G, W, su, sv) = block
    o = ref.block_pipeline(b["X"], b["G"], b["W"], b["sign_u"], b["sign_v"], spec, cfg.group, cfg.low_bits,
                           cfg.high_bits, cfg.budget, cfg.block, cfg.damp)
    assert o["bits"] == bits
    for name, grp, d_out, d_in in spec:
        p = q.pipes[name]
        What = torch.empty_like(W[name])
        K.kq_dequant_revert(p.codes, p.scale, p.zero, cfg.group, p.s_x, p.s_g, su[name], sv[name], What)
        torch.cuda.synchronize()
        HX = ref.accum_factor(b["X"][grp])
        HG = ref.accum_factor(b["G"][name])
        loss = ref.proxy_loss(b["W"][name], What.cpu().numpy(), HX, HG)
        want = o["layers"][name]["loss"]
        assert abs(loss - want) <= 1e-3 * want, (name, loss, want)
