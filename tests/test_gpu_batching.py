"""Graph workspace query and a short dynamic-batching run on the GPU."""
import numpy as np
import pytest
import torch

from paper_2511_19457_gb300 import batching as bt
from paper_2511_19457_gb300 import synth

pytestmark = pytest.mark.gpu


def test_graph_workspace_grows_with_batch_and_holds_activations():
    from paper_2511_19457_gb300 import sparoa as sp
    from paper_2511_19457_gb300 import calibrate as cal
    ctx = sp.Context(0)
    ops, _, _ = synth.resnet18(batch=1)
    graph = sp.Graph(ops)
    w = [sp.sparoa_graph_workspace(ctx, graph, (B, 224, 224, 3)) for B in (1, 2, 4)]
    # every value's bf16 activation lives in the workspace
    for B, bytes_ in zip((1, 2, 4), w):
        ins = cal.graph_input_shapes(ops, (B, 224, 224, 3))
        outs = ins[1:] + [(B, 1, 1, 1000)]
        act = sum(2 * int(np.prod(s)) for s in outs)
        assert act <= bytes_ <= 2 * act + (8 << 20)
    assert w[0] < w[1] < w[2]
    # affine in B up to alignment: the per-image share is constant
    assert abs((w[2] - w[1]) - 2 * (w[1] - w[0])) <= 64 * 1024
    # a bad list is rejected exactly as the walk would reject it
    bad = [dict(o) for o in ops]
    bad[3]["input"] = 10
    with pytest.raises(sp.SparoaError):
        sp.sparoa_graph_workspace(ctx, sp.Graph(bad), (1, 224, 224, 3))
    ctx.close()


def test_dynamic_batch_short_run():
    from paper_2511_19457_gb300 import sparoa as sp
    ctx = sp.Context(0)
    ops, _, _ = synth.resnet18(batch=1)
    graph = sp.Graph(ops)
    gen = torch.Generator(device="cuda").manual_seed(0)

    def latency(B):
        x = torch.randn(B, 224, 224, 3, device="cuda", generator=gen).to(torch.bfloat16)
        sp.sparoa_run_graph(ctx, graph, x)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        sp.sparoa_run_graph(ctx, graph, x)
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e-3

    memory = lambda B: sp.sparoa_graph_workspace(ctx, graph, (B, 224, 224, 3))
    tr = bt.dynamic_batch(latency, memory, 1, sparsity=0.0, intensity=0.0, b_max=8, max_iter=3,
                          mem_max=memory(4))
    assert 1 <= tr.batch <= 4
    assert all(memory(b) <= memory(4) for b, *_ , n in tr.steps if n != "gradient step")
    ctx.close()
