"""GPU parity of the online data-dependent rotation (Sec. 4.1, Eq. 4-5): x' = x . P . BlockDiag(U_b)
formed on the device for layers whose activations cannot take it upstream (layers that share an
input but fold different P and U_b, such as Q, K and V).

The kernel sums float32 products in a fixed order and rounds once to the activation dtype, the
oracle forms x' in float64: every kernel value lies within the float32 sum's error bound plus
half a step of the format of the float64 value, and almost all equal its rounding.  The whole
linear with the rotation set equals, bit for bit, the same layer without it run on the kernel's
x', and matches the oracle's composite linear within the output tolerance."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _factors(rng, N, K, block):
    w = (W.gaussian_weights(rng, N, K, 0.02) * rng.uniform(0.2, 4.0, K)[None, :]).astype(np.float32)
    perm, rot = Q.qvla_block_svd_rotation(w, Q.F32, N, K, block)
    return w, perm, rot


def _pack(w, had, perm, rot, block, xdt="f16", ydt="f16"):
    N, K = w.shape
    wq = np.zeros((N, K // 2), np.uint8)
    ws = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(w, Q.F32, N, K, rot=rot, rot_block=block, perm=perm, had_block=had, wq=wq, wscale=ws)
    return G.make_layer(wq, ws, had, xdt, ydt), wq, ws


def _rotate(layer, x):
    xg = x.to(G.DEV).contiguous()
    out = torch.full_like(xg, float("nan"))
    Q.qvla_online_rotate(layer, xg, x.shape[0], out, G.stream())
    Q.qvla_check_device(G.stream())
    return out.cpu()


@pytest.mark.parametrize("dt", ["f16", "bf16", "f32"])
@pytest.mark.parametrize("M,K,block", [(1, 512, 64), (50, 1024, 64), (130, 2048, 32), (64, 256, 16), (70, 1024, 64)])
def test_online_rotation_matches_oracle(dt, M, K, block):
    rng = np.random.default_rng(M + K + block)
    w, perm, rot = _factors(rng, 64, K, block)
    layer, _, _ = _pack(w, min(K, 512), perm, rot, block, dt, "bf16" if dt == "f32" else dt)
    Q.qvla_layer_set_online_rotation(layer, perm, rot, block)
    x = W.as_dtype(W.gaussian_with_outliers(rng, M, K, 5, 20.0), dt)
    got = _rotate(layer, x).double().numpy()
    xv = x.double().numpy()
    ref64 = O.upstream_activation_transform(xv, perm, rot, block)
    # error bound of the float32 sum of rot_block products (each rounded, then added in order)
    xp = np.abs(O.apply_permutation(xv, perm))
    mag = np.concatenate([xp[:, b * block:(b + 1) * block] @ np.abs(rot[b]) for b in range(K // block)], axis=1)
    bound = (block + 2) * 2.0 ** -24 * mag + 1e-30
    assert np.all(np.isfinite(got))
    if dt == "f32":
        assert np.all(np.abs(got - ref64) <= bound)
    else:
        # got is the rounding of a float32 sum within `bound` of the float64 value: at most half a
        # step of the format (at got) further away; equal to the oracle's rounding almost always
        half = 0.5 * np.maximum(G.ulp(got, dt), 2.0 ** -24 if dt == "f16" else 0.0)
        assert np.all(np.abs(got - ref64) <= bound + half * 1.0001)
        assert np.mean(got != O.round_to_format(ref64, dt)) < 0.02
    layer.close()


def test_linear_with_online_rotation():
    """The composite rotation of Sec. 4.1 with P and U_b applied online: equal to the plain layer on
    the kernel's x', within tolerance of the oracle, and an approximation of the float product."""
    rng = np.random.default_rng(41)
    M, N, K, block, had = 96, 384, 1024, 64, 512
    w, perm, rot = _factors(rng, N, K, block)
    x = W.as_dtype(W.gaussian_with_outliers(rng, M, K, 5, 20.0), "f16")
    online, wq, ws = _pack(w, had, perm, rot, block)
    Q.qvla_layer_set_online_rotation(online, perm, rot, block)
    got = G.linear(online, x, ydt="f16")
    x_rot = _rotate(online, x)
    plain, _, _ = _pack(w, had, perm, rot, block)
    assert np.array_equal(got, G.linear(plain, x_rot, ydt="f16"))
    _, oscale, codes = O.pack_weights(w.astype(np.float64), had, perm=perm, rot=rot, rot_block=block)
    ref = O.w4a4_linear(x_rot.double().numpy(), codes, oscale, had, out_fmt="f16")
    G.assert_output_close(got, ref["y"], "f16")
    exact = x.double().numpy() @ w.astype(np.float64).T
    assert O.relative_output_error(got, exact) < 0.35
    # the allocation-free linear takes the same path through its scratch
    y = torch.empty(M, N, dtype=torch.float16, device=G.DEV)
    Q.qvla_w4a4_linear_noalloc(online, x.to(G.DEV), M, -1, y, G.stream())
    Q.qvla_check_device(G.stream())
    assert np.array_equal(y.double().cpu().numpy(), got)
    # removing the rotation gives the plain layer back
    Q.qvla_layer_set_online_rotation(online, None, None, 0)
    assert np.array_equal(G.linear(online, x_rot, ydt="f16"), got)
    online.close()
    plain.close()


def test_shared_input_with_per_layer_rotations():
    """Q, K and V read one input but fold different P and U_b (chosen from their own weights):
    each layer rotates the shared x online, per step table included."""
    rng = np.random.default_rng(7)
    M, K, block, had = 50, 2048, 64, 2048
    x = W.as_dtype(W.gaussian_with_outliers(rng, M, K, 8, 20.0), "bf16")
    for n in (2048, 256, 256):
        w, perm, rot = _factors(rng, n, K, block)
        layer, wq, ws = _pack(w, had, perm, rot, block, "bf16", "bf16")
        Q.qvla_layer_set_online_rotation(layer, perm, rot, block)
        x_rot = _rotate(layer, x)
        table = O.calibrate_step_table([x_rot.double().numpy()], had)
        Q.qvla_set_step_scales(layer, table)
        _, oscale, codes = O.pack_weights(w.astype(np.float64), had, perm=perm, rot=rot, rot_block=block)
        for step in (-1, 0):
            got = G.linear(layer, x, step=step, ydt="bf16")
            ref = O.w4a4_linear(x_rot.double().numpy(), codes, oscale, had, table=table if step >= 0 else None,
                                step=step if step >= 0 else None, out_fmt="bf16")
            G.assert_output_close(got, ref["y"], "bf16")
        assert O.relative_output_error(got, x.double().numpy() @ w.astype(np.float64).T) < 0.35
        layer.close()


def test_online_rotation_rules():
    rng = np.random.default_rng(3)
    K, block = 512, 64
    w, perm, rot = _factors(rng, 64, K, block)
    layer, _, _ = _pack(w, 512, perm, rot, block)
    x = torch.zeros(4, K, dtype=torch.float16, device=G.DEV)
    out = torch.zeros_like(x)
    with pytest.raises(Q.QvlaError) as e:  # no rotation set yet
        Q.qvla_online_rotate(layer, x, 4, out, G.stream())
    assert e.value.status == 1
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_layer_set_online_rotation(layer, perm, np.zeros((K // 128, 128, 128)), 128)
    assert e.value.status == 2
    bad = perm.copy()
    bad[1] = bad[0]
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_layer_set_online_rotation(layer, bad, rot, block)
    assert e.value.status == 1
    Q.qvla_layer_set_online_rotation(layer, perm, None, 0)  # a permutation alone
    got = _rotate(layer, W.as_dtype(np.arange(4 * K, dtype=np.float32).reshape(4, K) % 97, "f16"))
    assert np.array_equal(got.numpy(), (np.arange(4 * K).reshape(4, K) % 97)[:, perm].astype(np.float16))
    Q.qvla_layer_set_online_rotation(layer, perm, rot, block)
    xq = torch.zeros(4, K // 2, dtype=torch.uint8, device=G.DEV)
    xs = torch.zeros(4, dtype=torch.float32, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_rotate_quantize(layer, x, 4, -1, xq, xs, None, G.stream())
    assert e.value.status == 2
    y = torch.zeros(4, 64, dtype=torch.float16, device=G.DEV)
    nb = Q.qvla_w4a8_workspace_bytes(layer, 4)
    work = torch.empty(nb, dtype=torch.uint8, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a8_linear(layer, x, 4, -1, y, work, nb, G.stream())
    assert e.value.status == 2
    layer.close()
