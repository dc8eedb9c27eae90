"""The seeded input generator, pinned against library routines and its stated distributions."""
import numpy as np
import pytest
import torch

import synth


def test_philox_matches_numpy_bit_generator():
    # numpy's Philox (4x64, 10 rounds) bumps its counter before producing a block,
    # so state counter c yields the block for counter c + 1.
    for key, ctr in [((7, 9), (5, 0, 0, 0)), ((0xDEADBEEF, 3), (2 ** 40, 1, 0, 0)), ((1, 2), (0, 0, 0, 7))]:
        g = np.random.Philox(counter=np.array(ctr, dtype=np.uint64), key=np.array(key, dtype=np.uint64))
        ref = g.random_raw(8)
        c = list(ctr)
        for blk in range(2):
            c[0] += 1
            assert list(synth.philox4x64_10(c, key)) == list(ref[4 * blk:4 * blk + 4])


def test_philox_random123_known_answer():
    # Known-answer vector of the Random123 distribution for philox4x64_10, counter 0 and key 0.
    out = synth.philox4x64_10([0, 0, 0, 0], [0, 0])
    assert [int(x) for x in out] == [0x16554D9ECA36314C, 0xDB20FE9D672D0FDC, 0xD7E772CEE186176B,
                                     0x7E68B68AEC7BA23B]


def test_normal_moments_and_bounds():
    x = synth.normal_f32(0, 123, 400_000, 0.02).astype(np.float64)
    assert abs(x.mean()) < 3 * 0.02 / np.sqrt(len(x)) * 2
    assert abs(x.std() / 0.02 - 1) < 5e-3
    # Irwin-Hall(8) support is +-4*sqrt(3/2) ... in std units: 4 / sqrt(8/12) = 4.899
    assert np.abs(x).max() <= 0.02 * 4.9


def test_bf16_is_round_to_nearest_even_of_the_f32_draw():
    f = synth.normal_f32(0, 77, 100_000, 0.02)
    b = synth.normal_bf16(0, 77, 100_000, 0.02)
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(b, ref)


def test_slices_regenerate_independently():
    full = synth.normal_bf16(3, 9, 1000, 0.02)
    part = synth.normal_bf16(3, 9, 300, 0.02, start=500)
    assert np.array_equal(full[500:800], part)


def test_zipf_rank_frequencies():
    v, s, n = 1000, 1.1, 200_000
    ids = synth.zipf_ids(1, 5, n, v, s)
    assert ids.min() >= 0 and ids.max() < v
    h = np.sum(np.arange(1, v + 1, dtype=np.float64) ** -s)
    for k in (1, 2, 10):
        expect = k ** -s / h
        got = np.mean(ids == k - 1)
        assert abs(got - expect) < 5 * np.sqrt(expect / n)


def test_uniform_ids_and_lengths():
    x = synth.uniform_int(1, 3, 100_000, 0, 4095)
    assert x.min() == 0 and x.max() == 4095
    assert abs(x.mean() - 2047.5) < 20
    w = synth.workload("7b_decode")
    lens = synth.prompt_lengths(w)
    assert lens.min() >= 1024 and lens.max() <= 2048 and len(lens) == 128


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_prompt_layout(name):
    w = synth.workload(name)
    inc, inc_off, cand, cand_off = synth.prompts(w, items=[0, 1])
    lens = synth.prompt_lengths(w)
    assert np.array_equal(np.diff(inc_off), [w.inc_len, w.inc_len])
    assert np.array_equal(np.diff(inc_off) + np.diff(cand_off), lens[:2])
    # the incumbent is shared by every item of the batch
    assert np.array_equal(inc[:w.inc_len], inc[w.inc_len:])
    assert inc.max() < w.model.vocab and cand.max() < w.model.vocab
