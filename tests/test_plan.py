"""Host logic of the C ABI, without a GPU: the GEMM tile planner and the
decode-attention chunk planner (gf_plan_gemm, gf_plan_decode_chunk).

The planner's choices must always satisfy what the GEMM kernel can run (a
swapped tile holds every activation row, split-K only with atomic
accumulation, each split at least four 64-column k-blocks), and they must
follow the stated rules: swap operands for decode-sized M, 256-wide tiles once
there are four 128-row blocks, SwiGLU above 64 rows on non-swapped tiles, and
about one wave of (tile, split) units for split-K.
"""
import itertools

import pytest

import paper_2605_31464_gb300 as gf
from paper_2605_31464_gb300 import _build

MODES = [gf.GF_GEMM_STORE_F32, gf.GF_GEMM_ADD_F32, gf.GF_GEMM_ATOMIC_F32, gf.GF_GEMM_STORE_BF16, gf.GF_GEMM_SWIGLU]
SMS = 152


@pytest.fixture(scope="module", autouse=True)
def _lib():
    _build.build()
    gf.load()


def plan(M, N, K, mode, sms=SMS):
    return gf.gf_plan_gemm(sms, M, N, K, mode)


# (N, K) of the 1.5B/7B/14B linears: QKV, O, gate/up (interleaved), down, LM head
SHAPES = [(2048, 1536), (1536, 1536), (17920, 1536), (1536, 8960), (151936, 1536),
          (4608, 3584), (3584, 3584), (37888, 3584), (3584, 18944), (152064, 3584),
          (7168, 5120), (5120, 5120), (27648, 5120), (5120, 13824), (152064, 5120)]
ROWS = [1, 2, 31, 32, 33, 63, 64, 65, 96, 127, 128, 129, 200, 384, 512, 513, 4096, 196608]


@pytest.mark.parametrize("mode", MODES)
def test_plans_are_runnable(mode):
    for (N, K), M in itertools.product(SHAPES, ROWS):
        p = plan(M, N, K, mode)
        bn, splits, swap = p["bn"], p["splits"], p["swap"]
        assert splits >= 1
        if splits > 1:
            assert mode == gf.GF_GEMM_ATOMIC_F32, (M, N, K, p)
            assert splits <= max(1, (K // 64) // 4), (M, N, K, p)
        if swap:
            assert M <= 128 and N % 32 == 0, (M, N, K, p)
            assert bn in (32, 64, 128) and bn >= M, (M, N, K, p)
            assert bn == min(b for b in (32, 64, 128) if b >= M), "the narrowest tile that holds every row"
            assert mode in (gf.GF_GEMM_STORE_F32, gf.GF_GEMM_ATOMIC_F32, gf.GF_GEMM_SWIGLU), (M, mode)
        else:
            assert bn in (64, 128, 256), (M, N, K, p)


@pytest.mark.parametrize("mode", MODES)
def test_plans_follow_the_rules(mode):
    for (N, K), M in itertools.product(SHAPES, ROWS):
        p = plan(M, N, K, mode)
        swappable = mode in (gf.GF_GEMM_STORE_F32, gf.GF_GEMM_ATOMIC_F32) or (mode == gf.GF_GEMM_SWIGLU and M <= 64)
        assert p["swap"] == (M <= 128 and swappable), (M, N, K, mode, p)
        if not p["swap"] and (M + 127) // 128 >= 4:
            assert p["bn"] == 256 and p["splits"] == 1, (M, N, K, mode, p)
        if mode == gf.GF_GEMM_SWIGLU and M > 64:
            assert not p["swap"] and p["bn"] == 256, (M, N, K, p)


def test_split_k_fills_about_one_wave():
    for (N, K), M in itertools.product(SHAPES, [1, 32, 64, 128]):
        p = plan(M, N, K, gf.GF_GEMM_ATOMIC_F32)
        assert p["swap"]
        tiles = (N + 127) // 128
        cap = max(1, (K // 64) // 4)
        if tiles >= SMS:
            assert p["splits"] == 1, (N, K, p)
        elif p["splits"] < cap:
            # nearest whole number of splits to one wave of (tile, split) units
            assert abs(tiles * p["splits"] - SMS) <= tiles / 2 + 1e-9, (N, K, p)


def test_decode_shapes_of_the_7b_model():
    # 32 sequences: every linear streams its weights as the 128-row operand
    assert plan(32, 4608, 3584, gf.GF_GEMM_ATOMIC_F32) == dict(bn=32, splits=4, swap=True)
    assert plan(32, 3584, 3584, gf.GF_GEMM_ATOMIC_F32) == dict(bn=32, splits=5, swap=True)
    assert plan(32, 37888, 3584, gf.GF_GEMM_SWIGLU) == dict(bn=32, splits=1, swap=True)
    assert plan(32, 3584, 18944, gf.GF_GEMM_ATOMIC_F32) == dict(bn=32, splits=5, swap=True)
    assert plan(32, 152064, 3584, gf.GF_GEMM_STORE_F32) == dict(bn=32, splits=1, swap=True)
    # 128 sequences: SwiGLU moves to non-swapped 256-wide tiles
    assert plan(128, 37888, 3584, gf.GF_GEMM_SWIGLU) == dict(bn=256, splits=1, swap=False)
    assert plan(128, 4608, 3584, gf.GF_GEMM_ATOMIC_F32)["swap"]


def test_prefill_shapes_use_full_width_tiles():
    for (N, K), mode in itertools.product(SHAPES, MODES):
        assert plan(196608, N, K, mode) == dict(bn=256, splits=1, swap=False)


def test_plan_depends_on_the_sm_count():
    few = plan(32, 4608, 3584, gf.GF_GEMM_ATOMIC_F32, sms=36)
    many = plan(32, 4608, 3584, gf.GF_GEMM_ATOMIC_F32, sms=152)
    assert few["splits"] == 1 and many["splits"] == 4


def test_bad_plan_arguments_are_refused():
    for args in [(0, 32, 4608, 3584, 0), (SMS, 0, 4608, 3584, 0), (SMS, 32, 0, 3584, 0), (SMS, 32, 4608, 0, 0),
                 (SMS, 32, 4608, 3584, -1), (SMS, 32, 4608, 3584, 5)]:
        with pytest.raises(gf.GfError) as e:
            gf.gf_plan_gemm(*args)
        assert e.value.code == gf.GF_EINVAL


def test_decode_chunk_is_the_longest_that_keeps_two_ctas_per_sm():
    for B, n_kv, ctx in itertools.product([1, 2, 8, 32, 128, 512], [1, 2, 4, 8], [1, 64, 1000, 2048, 6144, 16384]):
        c = gf.gf_plan_decode_chunk(B, n_kv, ctx, SMS)
        ctas = lambda chunk: B * n_kv * -(-ctx // chunk)
        assert c in (256, 512, 1024)
        if c > 256:
            assert ctas(c) >= 2 * SMS, (B, n_kv, ctx, c)
        if c < 1024:
            assert ctas(2 * c) < 2 * SMS, (B, n_kv, ctx, c)


def test_decode_chunk_of_the_benchmarked_batches():
    assert gf.gf_plan_decode_chunk(32, 4, 6144 + 256, SMS) == 1024    # 7B, 32 prompts of 6144
    assert gf.gf_plan_decode_chunk(8, 8, 16384 + 128, SMS) == 1024    # 14B, 8 prompts of 16384
    assert gf.gf_plan_decode_chunk(1, 1, 128, SMS) == 256
    with pytest.raises(gf.GfError):
        gf.gf_plan_decode_chunk(0, 4, 6144, SMS)
