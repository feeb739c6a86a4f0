"""Per-operator threshold calibration on this GPU.

The paper obtains its ground-truth thresholds offline, by an exhaustive grid
over sparsity and input size per operator, taking as the true threshold the
point where the faster device changes (Sec. 3.3).  The same acquisition on
one GB300: for each operator kind and size, the dense tensor-core kernel and
the zero-skip kernel are each forced and timed over a grid of activation
zero fractions rho, for unstructured and block-structured zeros.  The
calibrated sparsity threshold of that (kind, size, structure) is the
smallest grid rho from which zero-skip is faster at that rho and at every
larger one.  No grid rho qualifies: s_thr = 2 (never met, since zeros never
exceed numel).  It is stored as a table (JSON), and graphs take their
per-operator thresholds from the entry of the same kind nearest in FLOPs.

Calibrated thresholds set c_thr = 0: the second rule of Sec. 3 (dense but
light -> the CUDA-core side) is absorbed by the per-size measurement, since
an operator so light that zero-skip wins even at rho = 0 gets s_thr = 0.

Only ``calibrate`` touches the GPU; the table logic (crossover, lookup,
shape propagation, ``apply``) is host-side and runs anywhere.
"""
from __future__ import annotations

import json
import math
import os

TABLE_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "thresholds_gb300.json")
NEVER = 2.0  # an s_thr no zero fraction reaches

RHO_GRID = (0.0, 0.3, 0.5, 0.6, 0.7, 0.8, 0.9, 0.95)
STRUCTURES = ("unstructured", "block")

# Operator sizes of the calibration grid: the distinct conv / FC shapes of
# ResNet-18 at batch 8, MobileNetV2 at batch 32 and the 768 -> 3072 -> 768
# MLP down projection, plus the batch-32 3x3 64->64 conv.
# fc: (M, K, N); conv: (B, H, W, C_in, C_out, k, stride, pad).
DEFAULT_SPECS = (
    ("fc", (8, 512, 1000)), ("fc", (32, 1280, 1000)), ("fc", (64, 512, 512)),
    ("fc", (256, 3072, 768)), ("fc", (1024, 3072, 768)), ("fc", (4096, 3072, 768)),
    ("conv", (8, 56, 56, 64, 64, 3, 1, 1)), ("conv", (32, 56, 56, 64, 64, 3, 1, 1)),
    ("conv", (8, 28, 28, 128, 128, 3, 1, 1)), ("conv", (8, 14, 14, 256, 256, 3, 1, 1)),
    ("conv", (8, 7, 7, 512, 512, 3, 1, 1)),
    ("conv", (8, 56, 56, 64, 128, 3, 2, 1)), ("conv", (8, 28, 28, 128, 256, 3, 2, 1)),
    ("conv", (8, 14, 14, 256, 512, 3, 2, 1)),
    ("conv", (8, 56, 56, 64, 128, 1, 2, 0)), ("conv", (8, 28, 28, 128, 256, 1, 2, 0)),
    ("conv", (8, 14, 14, 256, 512, 1, 2, 0)),
    ("conv", (32, 56, 56, 144, 24, 1, 1, 0)), ("conv", (32, 56, 56, 24, 144, 1, 1, 0)),
    ("conv", (32, 28, 28, 192, 32, 1, 1, 0)), ("conv", (32, 14, 14, 384, 64, 1, 1, 0)),
    ("conv", (32, 14, 14, 576, 96, 1, 1, 0)), ("conv", (32, 14, 14, 96, 576, 1, 1, 0)),
    ("conv", (32, 7, 7, 960, 160, 1, 1, 0)), ("conv", (32, 7, 7, 320, 1280, 1, 1, 0)),
)


# ---------------------------------------------------------------------------
# host-side table logic
# ---------------------------------------------------------------------------
def kind_of(op: str, shape) -> str:
    """The calibration kind: FC with few rows (column-compacting kernel) and
    larger GEMMs are separate kinds; a conv's kind is its window and stride."""
    if op == "fc":
        return "fc_small" if shape[0] <= 128 else "gemm"
    k, s = shape[5], shape[6]
    return f"conv{k}x{k}s{s}"


def flops_of(op: str, shape) -> float:
    """Dense multiply-add FLOPs of one call (2 per MAC)."""
    if op == "fc":
        M, K, N = shape
        return 2.0 * M * K * N
    B, H, W, C, Co, k, s, p = shape
    Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
    return 2.0 * B * Ho * Wo * Co * C * k * k


def crossover(rhos, dense_us, skip_us) -> float:
    """Smallest grid rho from which zero-skip is faster at every larger grid
    rho (rhos ascending); NEVER when it is not faster at the largest one."""
    s_thr = NEVER
    for r, d, z in reversed(list(zip(rhos, dense_us, skip_us))):
        if not z < d:
            break
        s_thr = float(r)
    return s_thr


def thresholds_for(table: dict, op: str, shape, structure: str = "unstructured"):
    """Thresholds dict for one operator from the table entry of the same kind
    and structure nearest in log FLOPs, or None when the kind is absent."""
    kind = kind_of(op, shape)
    f = math.log(flops_of(op, shape))
    best = None
    for e in table.get("entries", ()):
        if e["kind"] != kind or e["structure"] != structure:
            continue
        d = abs(math.log(e["flops"]) - f)
        if best is None or d < best[0]:
            best = (d, e)
    if best is None:
        return None
    return {"s_thr": float(best[1]["s_thr"]), "c_thr": 0.0}


def graph_input_shapes(ops: list, x_shape) -> list:
    """NHWC shape of each operator's input value (value 0 = the graph input,
    j + 1 = output of op j), propagated through the operator list."""
    shapes = [tuple(x_shape)]
    ins = []
    for op in ops:
        B, H, W, C = shapes[op["input"]]
        ins.append((B, H, W, C))
        kind = op["kind"]
        if kind == "conv" or kind == "maxpool":
            k, s, p = op["k"], op["stride"], op["pad"]
            Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
            shapes.append((B, Ho, Wo, op["cout"] if kind == "conv" else C))
        elif kind == "avgpool":
            shapes.append((B, 1, 1, C))
        elif kind == "attention":
            shapes.append((B, H, W, C // 3))
        elif kind == "tokens":
            shapes.append((B, 1, H * W + 1, C))
        elif kind == "select":
            shapes.append((B, 1, 1, C))
        elif kind == "fc":
            shapes.append((B, 1, 1, op["cout"]))
        else:
            shapes.append((B, H, W, C))
    return ins


def apply(ops: list, x_shape, table: dict, structure: str = "unstructured") -> list:
    """A copy of a graph's operator list with each non-grouped conv and each
    FC given the calibrated thresholds of its kind and size.  The operator
    on the graph input (dense by construction) and kinds the table lacks
    keep theirs."""
    out = []
    for op, (B, H, W, C) in zip(ops, graph_input_shapes(ops, x_shape)):
        op = dict(op)
        t = None
        if op["kind"] == "fc":
            t = thresholds_for(table, "fc", (B, H * W * C, op["cout"]), structure)
        elif op["kind"] == "conv" and op.get("groups", 1) == 1 and op["input"] != 0:
            t = thresholds_for(table, "conv", (B, H, W, C, op["cout"], op["k"], op["stride"], op["pad"]),
                               structure)
        if t is not None:
            op["thr"] = dict(op.get("thr") or {}, **t)
        out.append(op)
    return out


def load_table(path: str | None = None) -> dict:
    with open(path or TABLE_PATH) as f:
        return json.load(f)


def summary(table: dict) -> dict:
    """{kind/structure: [(gflop, s_thr), ...]} for printing."""
    out = {}
    for e in table["entries"]:
        out.setdefault(f'{e["kind"]}/{e["structure"]}', []).append(
            (round(e["flops"] / 1e9, 3), e["s_thr"]))
    return out


# ---------------------------------------------------------------------------
# the measurement (GPU)
# ---------------------------------------------------------------------------
def calibrate(ctx, specs=DEFAULT_SPECS, rhos=RHO_GRID, structures=STRUCTURES, seed: int = 0,
              l2_bytes: float = 129e6, max_sets: int = 16, replays: int = 8, log=None) -> dict:
    """Time forced-dense and forced-zero-skip for every (spec, structure, rho)
    on the context's device and return the thresholds table.  Each point is
    a CUDA graph over rotating input/output sets totalling more than 3x L2,
    replayed ``replays`` times; the inputs' statistics are computed before
    capture (a graph receives them from the producer's epilogue)."""
    import torch

    from . import sparoa as sp
    from . import synth

    dev = torch.device("cuda", ctx.device)
    gen = torch.Generator(device=dev).manual_seed(seed)
    entries = []
    for op, shape in specs:
        shape = tuple(int(v) for v in shape)
        if op == "fc":
            M, K, N = shape
            w = (torch.randn(N, K, device=dev, generator=gen) / K ** 0.5).to(torch.bfloat16)
            w_kn = w.t().contiguous()
            x_shape, y_shape, occ_rc = (M, K), (M, N), (M, K)
            y_dtype = torch.float32 if M <= 128 else torch.bfloat16
        else:
            B, H, W, C, Co, k, s, p = shape
            w = (torch.randn(Co, k, k, C, device=dev, generator=gen) / (k * k * C) ** 0.5).to(torch.bfloat16)
            Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
            x_shape, y_shape, occ_rc = (B, H, W, C), (B, Ho, Wo, Co), (B * H * W, C)
            y_dtype = torch.bfloat16
        set_bytes = 2 * math.prod(x_shape) + y_dtype.itemsize * math.prod(y_shape)
        nb = max(2, min(max_sets, int(3 * l2_bytes / set_bytes) + 1))
        for structure in structures:
            dense_us, skip_us, measured = [], [], []
            for rho in rhos:
                xs = [synth.structured_activation(x_shape, rho, structure, gen, dev) for _ in range(nb)]
                ys = [torch.empty(*y_shape, dtype=y_dtype, device=dev) for _ in range(nb)]
                occ = [sp.OccupancyBuffer(*occ_rc) for _ in range(nb)]
                for j in range(nb):
                    st = sp.sparoa_op_stats(ctx, xs[j], x_shape, occ=occ[j], host=(j == 0))
                    if j == 0:
                        measured.append(round(float(st.sparsity), 4))

                def call(j, thr):
                    if op == "fc":
                        sp.sparoa_gemm(ctx, xs[j], w, ys[j], W_kn=w_kn, thr=thr, x_occ=occ[j])
                    else:
                        sp.sparoa_conv2d(ctx, xs[j], w, ys[j], stride=shape[6], pad=shape[7], thr=thr,
                                         act=sp.ACT_RELU, x_occ=occ[j])

                for force, acc in ((sp.PATH_DENSE, dense_us), (sp.PATH_SKIP, skip_us)):
                    thr = sp.thresholds(force_path=force)
                    for j in range(nb):
                        call(j, thr)
                    torch.cuda.synchronize(dev)
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(g):
                        for j in range(nb):
                            call(j, thr)
                    g.replay()
                    e0 = torch.cuda.Event(enable_timing=True)
                    e1 = torch.cuda.Event(enable_timing=True)
                    torch.cuda.synchronize(dev)
                    e0.record()
                    for _ in range(replays):
                        g.replay()
                    e1.record()
                    torch.cuda.synchronize(dev)
                    acc.append(round(e0.elapsed_time(e1) * 1e3 / (replays * nb), 3))
                    del g
                del xs, ys, occ
            e = {"op": op, "shape": list(shape), "kind": kind_of(op, shape), "structure": structure,
                 "flops": flops_of(op, shape), "rho": list(rhos), "measured_rho": measured,
                 "dense_us": dense_us, "skip_us": skip_us,
                 "s_thr": crossover(rhos, dense_us, skip_us), "rotating_sets": nb}
            entries.append(e)
            if log:
                log(e)
        torch.cuda.empty_cache()
    return {"device": torch.cuda.get_device_name(dev), "rho_grid": list(rhos),
            "structures": list(structures), "timing": f"CUDA graph of rotating sets > 3 x L2, "
                                                      f"{replays} replays, us per call",
            "entries": entries}
