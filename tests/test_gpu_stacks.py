"""GPU parity of whole layer stacks, run as the benchmark runs them (CUDA-graph replay of one
pass, 2 kernels per linear).

DiT action head (18 blocks, M = 50 tokens, T = 10 denoising steps): per-step scale tables
(Sec. 4.2, Eq. 6, per-tensor reading) calibrated by the oracle on a separate calibration draw,
then every linear of the stack checked against the oracle at the first, a middle and the last
step; the evaluation draw exceeds the calibrated peaks, so codes clamp at +-7.

Backbone (18 layers of hidden 2048, MLP 16384, per-token scales): the M = 816 prefix and an
M = 1 decode token, every linear checked on sampled rows (per-token quantisation makes each row
independent) and sampled output channels.

Each linear reads its own seeded input, drawn for both sides from the same generator."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import stack as S
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu

DIT_SEED, DIT_M, DIT_T, CAL_ROWS = 2, 50, 10, 16


def test_dit_stack_every_linear_at_three_steps():
    weights = W.dit_stack(DIT_SEED)
    tables = [O.calibrate_step_table([W.dit_layer_input(DIT_SEED + 1000, i, t, CAL_ROWS, w.k, DIT_T)
                                      for t in range(DIT_T)], w.had_block)
              for i, w in enumerate(weights)]
    st = S.LinearStack(weights, DIT_M, "f16", "f16", G.DEV)
    st.set_step_tables(tables)
    clamped = 0
    try:
        for t in (0, 4, DIT_T - 1):
            xs = [W.dit_layer_input(DIT_SEED, i, t, DIT_M, w.k, DIT_T) for i, w in enumerate(weights)]
            for i, x in enumerate(xs):
                st.set_input(i, torch.from_numpy(x))
            g = st.capture(t)
            for y in st.y:
                y.fill_(float("nan"))
            g.replay()
            torch.cuda.synchronize()
            G.Q.qvla_check_device(G.stream())
            for i, w in enumerate(weights):
                x16 = st.x[i].double().cpu().numpy()  # the fp16 values both sides quantise
                ref = O.w4a4_linear(x16, w.codes, w.wscale, w.had_block, bias=w.bias, table=tables[i], step=t,
                                    out_fmt="f16")
                clamped += int(np.count_nonzero(np.abs(ref["y_rot"]) > 7.5 * float(tables[i][t])))
                got = st.y[i].double().cpu().numpy()
                adj = G.assert_linear_close_modulo_ties(got, ref, w.codes, w.wscale, w.bias, "f16")
                assert np.mean(got == adj) > 0.98, w.name
    finally:
        st.close()
    assert clamped > 0, "the evaluation draw never exceeded the calibrated range"


def test_dit_stack_w4a8_every_linear():
    """The DiT stack with 8-bit activation codes (the appendix's W4A8 precision): per-step tables
    of absmax / 127 from the same calibration draw, every linear checked at the first and last
    step."""
    weights = W.dit_stack(DIT_SEED)
    tables = []
    for i, w in enumerate(weights):
        peaks = [O.robust_peak(O.rotate_activations(W.dit_layer_input(DIT_SEED + 1000, i, t, CAL_ROWS, w.k, DIT_T),
                                                    w.had_block)) for t in range(DIT_T)]
        tables.append(np.asarray(peaks, dtype=np.float32) / np.float32(127))
    st = S.LinearStack(weights, DIT_M, "f16", "f16", G.DEV, act_bits=8)
    st.set_step_tables(tables)
    try:
        for t in (0, DIT_T - 1):
            for i, w in enumerate(weights):
                st.set_input(i, torch.from_numpy(W.dit_layer_input(DIT_SEED, i, t, DIT_M, w.k, DIT_T)))
            g = st.capture(t)
            for y in st.y:
                y.fill_(float("nan"))
            g.replay()
            torch.cuda.synchronize()
            G.Q.qvla_check_device(G.stream())
            for i, w in enumerate(weights):
                ref = O.w4a4_linear(st.x[i].double().cpu().numpy(), w.codes, w.wscale, w.had_block, bias=w.bias,
                                    table=tables[i], step=t, out_fmt="f16", act_bits=8)
                G.assert_output_close(st.y[i].double().cpu().numpy(), ref["y"], "f16")
    finally:
        st.close()


def test_dit_stack_grouped_scales_every_linear():
    """The DiT stack in the paper's rotation configuration (Hadamard blocks of 64) with
    per-step, per-group tables over 128-channel groups, calibrated by the oracle on a separate
    16-token draw of channel-profiled inputs; every linear checked at the first and last step."""
    weights = W.dit_stack_blocks(W.dit_stack(DIT_SEED), 64)
    tables = [O.calibrate_step_table_grouped([W.dit_layer_input(DIT_SEED + 1000, i, t, CAL_ROWS, w.k, DIT_T, True)
                                              for t in range(DIT_T)], w.had_block)
              for i, w in enumerate(weights)]
    st = S.LinearStack(weights, DIT_M, "f16", "f16", G.DEV)
    st.set_step_tables(tables)
    try:
        for t in (0, DIT_T - 1):
            for i, w in enumerate(weights):
                st.set_input(i, torch.from_numpy(W.dit_layer_input(DIT_SEED, i, t, DIT_M, w.k, DIT_T, True)))
            g = st.capture(t)
            for y in st.y:
                y.fill_(float("nan"))
            g.replay()
            torch.cuda.synchronize()
            G.Q.qvla_check_device(G.stream())
            for i, w in enumerate(weights):
                ref = O.grouped_linear(st.x[i].double().cpu().numpy(), w.codes, w.wscale, w.had_block, tables[i], t,
                                       bias=w.bias, out_fmt="f16")
                G.assert_output_close(st.y[i].double().cpu().numpy(), ref["y"], "f16")
    finally:
        st.close()


def _backbone_check(weights, st, rows, seed):
    """Sampled rows of every linear; all output channels of qkv and o, 256 of down, 128 hidden
    units (gate and up rows) of the gated layer.  The oracle unpacks the sampled weight rows."""
    rng = np.random.default_rng(seed)
    ri = torch.as_tensor(rows, device=G.DEV)
    for i, w in enumerate(weights):
        x = st.x[i][ri].double().cpu().numpy()
        got = st.y[i][ri].double().cpu().numpy()
        if w.gated:
            units = np.sort(rng.choice(w.n, 128, replace=False))
            gate = O.w4a4_linear(x, O.unpack_int4(w.packed[units]), w.wscale[units], w.had_block, out_fmt="bf16")["y"]
            up = O.w4a4_linear(x, O.unpack_int4(w.packed[w.n + units]), w.wscale[w.n + units], w.had_block,
                               out_fmt="bf16")["y"]
            ref = O.round_to_format(O.gated_glue(gate, up), "bf16")
            G.assert_output_close(got[:, units], ref, "bf16")
        else:
            cols = np.arange(w.n) if w.k <= 2048 else np.sort(rng.choice(w.n, 256, replace=False))
            ref = O.w4a4_linear(x, O.unpack_int4(w.packed[cols]), w.wscale[cols], w.had_block, out_fmt="bf16")["y"]
            G.assert_output_close(got[:, cols], ref, "bf16")


@pytest.mark.parametrize("m", [816, 1])
def test_backbone_stack_sampled(m):
    weights = W.backbone_stack(seed=3)
    st = S.LinearStack(weights, m, "bf16", "bf16", G.DEV)
    try:
        for i, w in enumerate(weights):
            st.set_input(i, torch.from_numpy(W.backbone_layer_input(3, i, m, w.k)))
        g = st.capture(-1)
        for y in st.y:
            y.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        G.Q.qvla_check_device(G.stream())
        rows = np.sort(np.random.default_rng(m).choice(m, min(m, 4), replace=False))
        _backbone_check(weights, st, rows, seed=m + 1)
    finally:
        st.close()
