"""Shared checks for the GPU parity tests."""
import numpy as np

# Float tolerance of the path (bf16 inputs, fp32 accumulation):
#   max |err| <= 2e-2 * max |ref|  and  ||err||_F <= 5e-3 * ||ref||_F
MAX_REL = 2e-2
FRO_REL = 5e-3


def assert_close(got, ref, max_rel=MAX_REL, fro_rel=FRO_REL, what=""):
    got = np.asarray(got, dtype=np.float64).reshape(-1)
    ref = np.asarray(ref, dtype=np.float64).reshape(-1)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    scale = np.abs(ref).max()
    err = np.abs(got - ref)
    if scale == 0:
        assert err.max() == 0, f"{what}: expected all zeros, max |got| = {err.max()}"
        return
    assert err.max() <= max_rel * scale, f"{what}: max err {err.max():.3e} vs {max_rel}*{scale:.3e}"
    fro = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-300)
    assert fro <= fro_rel, f"{what}: relative Frobenius error {fro:.3e}"


def assert_occ_equal(occ_dev: dict, st, what=""):
    """Device occupancy block == oracle stats, bit for bit."""
    assert occ_dev["nnz"] == st.nnz, f"{what}: nnz {occ_dev['nnz']} != {st.nnz}"
    assert np.array_equal(occ_dev["col_nnz"], st.col_nnz), f"{what}: col_nnz"
    assert np.array_equal(occ_dev["tile_nnz"], st.tile_nnz), f"{what}: tile_nnz"
    assert np.array_equal(occ_dev["row_bm"], st.row_bm), f"{what}: row_bm"
    assert np.array_equal(occ_dev["blk_mask"], st.blk_mask), f"{what}: blk_mask"


def perturbed_chain_error(ops, x_bits, shape, ref_last_f64, rel=2.0 ** -24, seed=1):
    """Sensitivity of a graph's chained output to the smallest rounding error
    any fp32 kernel makes.  The oracle walks the graph again, but every
    operator's fp64 output is multiplied by (1 + u * rel), u ~ U(-1, 1) per
    element (rel = 2^-24: at most one fp32 rounding of the result), before
    the bf16 rounding that stores it.  Returns (max |err| / max |ref|,
    relative Frobenius error) of that walk's bf16 output against
    ``ref_last_f64``, the unperturbed walk's fp64 output of the last operator."""
    from oracle import oracle as orc
    rng = np.random.default_rng(seed)
    values = {0: (np.asarray(x_bits), tuple(shape))}
    last = None
    for i, op in enumerate(ops):
        xin, xs = values[op["input"]]
        res = values[op["residual"]][0] if op.get("residual", -1) >= 0 else None
        r = orc.run_op(op, xin, xs, res)
        y = r.out_f64 * (1.0 + rel * rng.uniform(-1.0, 1.0, size=r.out_f64.shape))
        bits = orc.f64_to_bf16(y).reshape(r.out_shape)
        values[i + 1] = (bits, r.out_shape)
        last = bits
    got = ((np.asarray(last, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)
           .astype(np.float64).reshape(-1))
    ref = np.asarray(ref_last_f64, dtype=np.float64).reshape(-1)
    err = np.abs(got - ref)
    return err.max() / np.abs(ref).max(), np.linalg.norm(got - ref) / np.linalg.norm(ref)
