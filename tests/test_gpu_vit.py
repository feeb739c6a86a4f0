"""Vision-transformer operators and a ViT-shaped graph against the oracle (GPU)."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth
from tests._parity import assert_close, assert_occ_equal

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2511_19457_gb300 import sparoa
    return sparoa


@pytest.fixture(scope="module")
def ctx(sp):
    c = sp.Context(0)
    yield c
    c.close()


def _rand_bits(shape, seed, scale=1.0, shift=0.0):
    g = torch.Generator().manual_seed(seed)
    return synth.to_bf16_bits(shift + scale * torch.randn(*shape, generator=g))


@pytest.mark.parametrize("R,C,affine", [(300, 768, True), (197, 64, False), (1, 8, True), (4099, 192, True),
                                         (7, 1024, True),    # longest row held in registers
                                         (5, 1032, True),    # re-read path
                                         (6304, 768, True),  # ViT-B/16 at batch 32
                                         (100000, 64, False)])  # several 128-row blocks per CTA
def test_layernorm(sp, ctx, R, C, affine):
    """Constant rows (every fourth) normalise to exact zeros without an affine,
    so the output's row bitmaps, block masks and counts see zero rows too."""
    xb = _rand_bits((R, C), R + C, 2.0, 1.0)
    xb.reshape(R, C)[::4] = xb.reshape(R, C)[::4, :1]
    gb = None
    if affine:
        g = torch.Generator().manual_seed(7)
        gb = np.stack([1 + 0.1 * torch.randn(C, generator=g).numpy(),
                       0.1 * torch.randn(C, generator=g).numpy()]).astype(np.float32)
    x = sp.bits_to_device(xb).view(R, C)
    y = torch.empty(R, C, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(R, C)
    sp.sparoa_layernorm(ctx, x, y, gamma_beta=None if gb is None else torch.from_numpy(gb).cuda(),
                        eps=1e-6, y_occ=yo)
    torch.cuda.synchronize()
    ref = orc.layernorm(xb, R, C, gb, 1e-6)
    ybits = sp.device_to_bits(y)
    assert_close(synth.bits_to_f32(ybits).astype(np.float64).reshape(R, C), ref, what=f"layernorm {R}x{C}")
    assert_occ_equal(yo.to_host(), orc.stats(ybits, R, C), "layernorm y_occ")


@pytest.mark.parametrize("N,T,heads,hd", [(2, 197, 12, 64), (1, 17, 3, 64), (3, 50, 4, 32), (1, 1, 1, 16),
                                          (1, 512, 2, 64), (2, 64, 2, 16), (1, 200, 2, 32)])
def test_attention(sp, ctx, N, T, heads, hd):
    D = heads * hd
    qkvb = _rand_bits((N, T, 3 * D), N * T + D)
    qkv = sp.bits_to_device(qkvb).view(N, T, 3 * D)
    y = torch.empty(N, T, D, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(N * T, D)
    sp.sparoa_attention(ctx, qkv, y, heads, y_occ=yo)
    torch.cuda.synchronize()
    ref = orc.attention(qkvb, N, T, heads, hd)
    ybits = sp.device_to_bits(y)
    assert_close(synth.bits_to_f32(ybits).astype(np.float64).reshape(N, T, D), ref,
                 what=f"attention N{N} T{T} h{heads} hd{hd}")
    assert_occ_equal(yo.to_host(), orc.stats(ybits, N * T, D), "attention y_occ")


def test_attention_rejects_unsupported(sp, ctx):
    qkv = torch.zeros(1, 600, 3 * 64, dtype=torch.bfloat16, device="cuda")
    y = torch.empty(1, 600, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sp.SparoaError):
        sp.sparoa_attention(ctx, qkv, y, 1)


@pytest.mark.parametrize("force", [1, 2])
def test_gelu_epilogue(sp, ctx, force):
    M, K, N = 197, 768, 3072
    xb = _rand_bits((M, K), 3)
    g = torch.Generator().manual_seed(4)
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / np.sqrt(K))
    bias = (0.02 * torch.randn(N, generator=g)).numpy().astype(np.float32)
    x = sp.bits_to_device(xb).view(M, K)
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    sp.sparoa_gemm(ctx, x, sp.bits_to_device(wb).view(N, K), y, bias=torch.from_numpy(bias).cuda(),
                   act=sp.ACT_GELU, thr=sp.thresholds(force_path=force))
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(0).choice(M, 48, replace=False))
    ref = orc.fc(xb.reshape(M, K)[rows], len(rows), K, wb, N, bias=bias, act=orc.ACT_GELU)
    assert_close(y.float().cpu().numpy().astype(np.float64)[rows], ref, what="gelu epilogue")


def _run_graph(sp, ops, xb, shape):
    ctx = sp.Context(0)
    graph = sp.Graph(ops)
    x = sp.bits_to_device(xb).view(*shape)
    recs = sp.sparoa_run_graph(ctx, graph, x, records=True)
    torch.cuda.synchronize()
    outs, occs = [], []
    for r in recs:
        shp = tuple(int(v) for v in r.out_shape)
        t = sp.view_device(r.output, (int(np.prod(shp)),))
        outs.append((sp.device_to_bits(t), shp))
        occs.append(sp.record_occupancy(r))
    ctx.close()
    return recs, outs, occs


def test_small_vit_teacher_forced(sp):
    """Every operator of a 2-layer ViT (64x64 input, 16 patches + class token,
    dim 192, 3 heads, MLP 768, GELU) on exactly the tensor the GPU fed it."""
    from tests.test_gpu_graph import _teacher_check
    ops, xb, shape = synth.vit(batch=2, img=64, dim=192, depth=2, heads=3, mlp=768, classes=16)
    recs, outs, occs = _run_graph(sp, ops, xb, shape)
    assert len(recs) == len(ops)
    _teacher_check(sp, ops, xb, shape, recs, outs, occs)
    kinds = {op["kind"] for op in ops}
    assert {"layernorm", "attention", "tokens", "select", "conv", "fc"} <= kinds


def test_small_vit_relu_mlp_dispatch(sp):
    """With ReLU MLPs (act = 1) the second MLP layer's input is about half
    zeros: the rule's decisions match the oracle's on it."""
    from tests.test_gpu_graph import _teacher_check
    ops, xb, shape = synth.vit(batch=1, img=64, dim=192, depth=1, heads=3, mlp=768, classes=16, act=1)
    recs, outs, occs = _run_graph(sp, ops, xb, shape)
    _teacher_check(sp, ops, xb, shape, recs, outs, occs)
    fc2 = [i for i, op in enumerate(ops) if op["kind"] == "conv" and op["cin"] == 768][0]
    assert 0.3 < recs[fc2].stats.sparsity < 0.7


def test_vit_b16_runs(sp):
    """ViT-B/16 at batch 1 through the walk: 197 tokens, 12 layers; the
    chained logits are compared with the oracle's chained walk loosely."""
    ops, xb, shape = synth.vit(batch=1)
    recs, outs, occs = _run_graph(sp, ops, xb, shape)
    assert outs[-1][1] == (1, 1, 1, 1000)
    logits = synth.bits_to_f32(outs[-1][0]).astype(np.float64)
    assert np.all(np.isfinite(logits))
    ref = orc.run_graph(ops, xb, shape)
    assert_close(logits, ref[-1].out_f64.reshape(-1), max_rel=8e-2, fro_rel=3e-2, what="vit-b16 chained logits")
