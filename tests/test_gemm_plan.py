"""CPU tests of the token-major GEMM's launch plan (Sec. 4.2, Eq. 7): the tile shape and the split
of K that qvla_w4a4_linear's GEMM takes for M > 128 tokens, read through qvla_debug_gemm_plan
(host logic only, no GPU).

The plan is a launch-time estimate fitted to GB300 measurements; these tests pin the decisions the
measurements justified and the rules around them:
  * the backbone's down projection (816 x 16384 -> 2048) runs 256 x 256 CTA pairs with each tile's
    K in 2 work units (43.3 us against 53.9 us for its best whole-tile shape);
  * 256 x 16384 -> 2048 runs 128 x 128 single CTAs in 4 units (26.6 against 53.8 us);
  * gated layers never split (their epilogue pairs gate and up columns of one accumulator);
  * without the workspace room for the partials every launch runs whole tiles;
  * a unit keeps at least 16 k-blocks, and a split is taken only where it is estimated 10% faster;
  * launches whose tiles already fill the SMs run whole tiles."""

import pytest

from paper_2605_28803_gb300 import qvla as Q

SMS = 152  # GB300


def plan(M, K, N, gated=False, room=True, sms=SMS):
    return Q.qvla_debug_gemm_plan(M, K, N, gated=gated, num_sms=sms, split_room=room)


def test_down_projection_runs_pairs_in_two_parts():
    assert plan(816, 16384, 2048) == ("pair 256x256", 2)


def test_few_token_tiles_split_in_four():
    assert plan(256, 16384, 2048) == ("single 128x128", 4)
    assert plan(150, 16384, 2048) == ("single 128x128", 4)  # a ragged token tile


def test_ragged_shapes_of_the_split_tests():
    # the shapes tests/test_gpu_split_k.py runs bit-identical against whole tiles
    assert plan(300, 16384, 2000) == ("single 128x256", 4)
    assert plan(700, 16384, 1904) == ("pair 256x256", 2)


def test_gated_layers_never_split():
    # the backbone's gate/up projection: 2 x 16384 weight rows
    assert plan(816, 2048, 32768, gated=True) == ("pair 256x256", 1)
    for M in (129, 256, 816):
        assert plan(M, 16384, 2048, gated=True)[1] == 1


@pytest.mark.parametrize("M,K,N", [(816, 16384, 2048), (256, 16384, 2048), (300, 16384, 2000), (700, 16384, 1904)])
def test_no_room_means_whole_tiles(M, K, N):
    shape, parts = plan(M, K, N, room=False)
    assert parts == 1
    assert shape == "single 128x128"  # the whole-tile choice at these sizes


def test_units_keep_sixteen_k_blocks():
    # K = 2048 has 16 k-blocks: no unit of 8
    assert plan(816, 2048, 2048)[1] == 1
    assert plan(256, 2048, 2048)[1] == 1
    # K = 4096 (32 k-blocks) could split in 2, but the estimate gains less than 10% there
    assert plan(150, 4096, 2048)[1] == 1


def test_full_waves_run_whole_tiles():
    for M, K, N in [(3200, 16384, 2048), (8192, 16384, 2048), (8192, 2048, 16384), (3200, 1024, 4096)]:
        assert plan(M, K, N)[1] == 1


def test_fewer_sms_change_the_plan_not_its_rules():
    # on a device with half the SMs the down projection's 32 pair tiles fill 38 pairs whole
    assert plan(816, 16384, 2048, sms=76)[1] == 1
    for M, K, N in [(816, 16384, 2048), (256, 16384, 2048), (150, 16384, 2048)]:
        for sms in (76, 132, 152, 160):
            shape, parts = plan(M, K, N, sms=sms)
            assert parts in (1, 2, 4)
            assert 16384 // 128 // parts >= 16


def test_plan_refuses_bad_arguments():
    for args in [(128, 1024, 1024), (816, 1000, 1024), (816, 1024, 1000), (816, 1024, 1024 + 128)]:
        gated = args == (816, 1024, 1024 + 128)
        with pytest.raises(Q.QvlaError) as e:
            plan(*args, gated=gated)
        assert e.value.status == 1
    with pytest.raises(Q.QvlaError):
        plan(816, 1024, 1024, sms=1)
