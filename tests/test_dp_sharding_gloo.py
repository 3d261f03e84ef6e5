"""Data-parallel sharding of the layer step over samples, on CPU with world_size-2 `gloo` ranks.

Each rank owns a contiguous block of samples (rows of X and gY).  The forward product and the
grad_input side of SCQ (per-sample scales, Sec. 5.3) need nothing from other ranks.  The step is
the same as on one device, bit for bit, with these exact exchanges:

  1. all-gather the per-sample zero points and ranges (Sec. 5.2 needs every group's range to
     water-fill the keep probabilities, so every rank draws the same p^ and kept set);
  2. all-reduce MIN / MAX of the per-channel minima and maxima before PCQ (Sec. 5.3: the
     per-channel scales span all samples);
  3. all-reduce SUM of the integer grad_weight accumulators (exact, any order), together with
     the column sums of sign(X) that its dequantization adds (one buffer).

Stochastic rounding takes its counter from the global element index (reading R5), so the codes
do not depend on the split.  The per-rank arithmetic is the oracle's (`oracle/method.py`); the
exchanges are torch.distributed collectives.  On the GPU the same exchanges would be NCCL
collectives on the range keys and int32 accumulators; every run here has one GPU, so that path
is not built and this test is its only check.
"""
import os
import socket
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
dist = pytest.importorskip("torch.distributed")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

f32 = np.float32


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _all_gather_rows(a):
    t = torch.from_numpy(np.ascontiguousarray(a))
    parts = [torch.empty_like(t) for _ in range(dist.get_world_size())]
    dist.all_gather(parts, t)
    return torch.cat(parts).numpy()


def _all_reduce(a, op):
    t = torch.from_numpy(np.ascontiguousarray(a))
    dist.all_reduce(t, op=op)
    return t.numpy()


def sharded_backward(om, g_loc, row0, M, rpg, sx_loc, sw, bits_s, mode_s, seed_s, bits_c, mode_c, seed_c):
    """SCQ backward of one rank's rows [row0, row0 + rows) of G = gY (.) Gamma.

    Returns the local PSQ branch (kept ids global, codes of this rank's kept samples), the
    grad_input accumulators and dequantized rows of this rank's samples, and the grad_weight
    accumulators and dW, which every rank ends with in full."""
    rows, D = g_loc.shape
    # exchange 1: the sample ranges of every rank, in global sample order
    z_loc, r_loc = om.sample_ranges(g_loc, rpg)
    z_s = _all_gather_rows(z_loc)
    r_s = _all_gather_rows(r_loc)
    # exchange 2: the channel minima and maxima over all samples
    z_c = _all_reduce(g_loc.min(axis=0).astype(f32), dist.ReduceOp.MIN)
    mx_c = _all_reduce(g_loc.max(axis=0).astype(f32), dist.ReduceOp.MAX)
    r_c = (mx_c - z_c).astype(f32)
    # the selection is a pure function of the global ranges: identical on every rank
    kept_s, ph_s, _ = om.select_groups(r_s, bits_s, mode_s, seed_s, om.STREAM_SEL_SAMPLE)
    kept_c, ph_c, _ = om.select_groups(r_c, bits_c, mode_c, seed_c, om.STREAM_SEL_CHANNEL)
    sc_s, ze_s = om.group_scale(r_s[kept_s], z_s[kept_s], ph_s[kept_s], bits_s)
    sc_c, ze_c = om.group_scale(r_c[kept_c], z_c[kept_c], ph_c[kept_c], bits_c)
    # PSQ on this rank's kept samples, SR counters at the global element index m D + j
    g0, g1 = row0 // rpg, (row0 + rows) // rpg
    mine = [(slot, gid) for slot, gid in enumerate(kept_s) if g0 <= gid < g1]
    cs_w = sw.astype(np.int64).sum(axis=0)
    K = sw.shape[1]
    dx_loc = np.zeros((rows, K), dtype=f32)
    acc_dx = []
    for slot, gid in mine:
        r = np.arange(gid * rpg, (gid + 1) * rpg)
        flat = r[:, None].astype(np.uint64) * np.uint64(D) + np.arange(D, dtype=np.uint64)[None, :]
        q = om.sr_codes(g_loc[r - row0], z_s[gid], r_s[gid], bits_s, seed_s, om.STREAM_SR_PSQ, flat)
        a = om.int_matmul(q, sw.T)
        acc_dx.append(a)
        dx_loc[r - row0] = om.dequant(sc_s[slot], a, ze_s[slot], cs_w[None, :])
    # PCQ on this rank's rows of every kept channel, counters at the global index j M + m
    m_glob = np.arange(row0, row0 + rows, dtype=np.uint64)
    flat = kept_c.astype(np.uint64)[:, None] * np.uint64(M) + m_glob[None, :]
    qc = om.sr_codes(g_loc[:, kept_c].T, z_c[kept_c][:, None], r_c[kept_c][:, None], bits_c, seed_c,
                     om.STREAM_SR_PCQ, flat)
    part = om.int_matmul(qc, sx_loc.T)                       # [kept channels, K] partial sums
    cs_x_part = sx_loc.astype(np.int64).sum(axis=0)          # [K] partial column sums
    # exchange 3: one integer all-reduce of the accumulators and the column sums
    red = _all_reduce(np.concatenate([part.reshape(-1), cs_x_part]).astype(np.int64), dist.ReduceOp.SUM)
    acc_dw = red[:part.size].reshape(part.shape)
    cs_x = red[part.size:]
    dw = np.zeros((sw.shape[0], K), dtype=f32)
    for s, j in enumerate(kept_c):
        dw[j] = om.dequant(sc_c[s], acc_dw[s], ze_c[s], cs_x)
    return dict(kept_s=kept_s, ph_s=ph_s, kept_c=kept_c, ph_c=ph_c, dx_loc=dx_loc, acc_dw=acc_dw, dw=dw,
                acc_dx=np.concatenate(acc_dx) if acc_dx else np.zeros((0, K), np.int64))


def _worker(rank, world, port, out_dir, kind):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import method as om
        from paper_2408_14267_gb300 import workloads as wl
        if kind == "linear":
            w = wl.sweep_point(64, 96, 40, 16, 4, seed=9, qseed=11)
            N = 16
            n_loc = N // world
            rpg = w["rows_per_group"]
            x_loc = w["x"][rank * n_loc * rpg:(rank + 1) * n_loc * rpg]
            sx_loc = om.sign(x_loc)
            wmat = w["w"]
        else:
            w = wl.conv_layer("dp conv", 8, 5, 6, 6, 7, 3, 1, 1, 2, 21, 31, sample_sigma=1.5)
            N, C, H, W = w["x"].shape
            n_loc = N // world
            x_loc = w["x"][rank * n_loc:(rank + 1) * n_loc]
            Ho, Wo = om.conv_out_hw(H, W, 3, 3, w["stride"], w["pad"])
            rpg = Ho * Wo
            sx_loc = om.sign(om.unfold(x_loc, 3, 3, w["stride"], w["pad"]))
            wmat = w["w"].reshape(w["w"].shape[0], -1)
        M = N * rpg
        row0 = rank * n_loc * rpg
        gy_loc = w["gy"][row0:row0 + n_loc * rpg]
        # forward: local rows only
        acc_y = om.int_matmul(sx_loc, om.sign(wmat))
        y_loc = (np.asarray(w["gamma"], f32)[None, :] * acc_y.astype(f32)).astype(f32)
        g_loc = om.grad_to_quantize(gy_loc, w["gamma"])
        out = sharded_backward(om, g_loc, row0, M, rpg, sx_loc, om.sign(wmat), w["bits_s"], w["mode_s"],
                               w["seed_s"], w["bits_c"], w["mode_c"], w["seed_c"])
        np.savez(os.path.join(out_dir, f"{kind}_rank{rank}.npz"), y_loc=y_loc, **out)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("kind", ["linear", "conv"])
def test_sharded_step_equals_single_rank(tmp_path, kind):
    from oracle import method as om
    from paper_2408_14267_gb300 import workloads as wl
    world = 2
    torch.multiprocessing.spawn(_worker, args=(world, _free_port(), str(tmp_path), kind), nprocs=world, join=True)
    r = [dict(np.load(tmp_path / f"{kind}_rank{i}.npz")) for i in range(world)]
    if kind == "linear":
        w = wl.sweep_point(64, 96, 40, 16, 4, seed=9, qseed=11)
        ref = om.layer_step_linear(w["x"], w["w"], w["gamma"], w["gy"], w["bits_s"], w["mode_s"], w["seed_s"],
                                   w["bits_c"], w["mode_c"], w["seed_c"], w["rows_per_group"])
        dx_ref = ref["dx"]
    else:
        w = wl.conv_layer("dp conv", 8, 5, 6, 6, 7, 3, 1, 1, 2, 21, 31, sample_sigma=1.5)
        ref = om.layer_step_conv(w["x"], w["w"], w["gamma"], w["gy"], w["stride"], w["pad"], w["bits_s"],
                                 w["mode_s"], w["seed_s"], w["bits_c"], w["mode_c"], w["seed_c"])
        # the sharded ranks return dX_u rows; fold the 1-rank unfolded rows the same way
        dx_ref = None
    # every rank drew the same selection as the single rank
    for x in r:
        assert np.array_equal(x["kept_s"], ref["psq"]["kept"]) and np.array_equal(x["ph_s"], ref["psq"]["p_hat"])
        assert np.array_equal(x["kept_c"], ref["pcq"]["kept"]) and np.array_equal(x["ph_c"], ref["pcq"]["p_hat"])
        # grad_weight: the all-reduced accumulators and dW equal the single rank's, bit for bit
        assert np.array_equal(x["acc_dw"], ref["acc_dw"])
        assert np.array_equal(x["dw"].reshape(ref["dw"].shape), ref["dw"])
    # forward and grad_input: the ranks' rows, concatenated, are the single rank's
    assert np.array_equal(np.concatenate([x["y_loc"] for x in r]), ref["y"])
    assert np.array_equal(np.concatenate([x["acc_dx"] for x in r]), ref["acc_dx"])
    if dx_ref is not None:
        assert np.array_equal(np.concatenate([x["dx_loc"] for x in r]), dx_ref)
    # the split is not trivial: both ranks kept some samples
    n_s = len(ref["psq"]["p_hat"])
    kept = ref["psq"]["kept"]
    assert (kept < n_s // 2).any() and (kept >= n_s // 2).any()
