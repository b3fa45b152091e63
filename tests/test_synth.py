"""The seeded input generator: definition, determinism, moments, bf16 rounding."""
import numpy as np
import torch

from wm_synth import configs, gen, inputs


def test_splitmix64_reference_sequence():
    # SplitMix64 seeded with state 0 (Vigna's reference generator): first outputs
    z = gen.mix64(np.arange(1, 4, dtype=np.uint64) * gen.GAMMA)
    assert [int(v) for v in z] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_values_are_deterministic_and_sliceable():
    a = gen.values("f32", 3, 7, 0, 1000)
    b = gen.values("f32", 3, 7, 400, 100)
    assert np.array_equal(a[400:500], b)
    idx = np.array([999, 0, 123], dtype=np.uint64)
    assert np.array_equal(gen.values_at("f32", 3, 7, idx), a[[999, 0, 123]])
    assert not np.array_equal(a, gen.values("f32", 4, 7, 0, 1000))


def test_moments_and_scaling():
    v = gen.values("f32", 0, 1, 0, 1 << 20).astype(np.float64)
    assert abs(v.mean()) < 5e-3 and abs(v.std() - 1.0) < 5e-3
    w = gen.values("f32", 0, 1, 0, 1 << 16, std=0.25, mean=1.0).astype(np.float64)
    assert abs(w.mean() - 1.0) < 5e-3 and abs(w.std() - 0.25) < 5e-3
    ones = gen.values("f32", 0, 1, 0, 100, std=0.0, mean=1.0)
    assert np.all(ones == 1.0)


def test_bf16_rounding_matches_torch_round_to_nearest_even():
    x = np.concatenate([gen.values("f32", 1, 2, 0, 100000, std=10.0),
                        np.array([0.0, -0.0, 1.0, 65504.0, 1e-40, 3.0e38], np.float32)])
    mine = gen.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(mine, ref)


def test_problem_paging_is_a_partition():
    for name in ("tiny_f32", "compress50", "large"):
        p = inputs.make_problem(configs.get(name), seed=0)
        used = p.page_table[p.page_table >= 0]
        assert np.array_equal(np.sort(used), np.arange(p.num_pages))
        for b, S in enumerate(p.seq_lens):
            n = int((p.page_table[b] >= 0).sum())
            assert n * p.w.page >= S + 1 > (n - 1) * p.w.page
    w = configs.get("large")
    p = inputs.make_problem(w, seed=0)
    assert p.seq_lens.min() >= w.ctx_lo and p.seq_lens.max() <= w.ctx


def test_chunked_generation_equals_the_one_pass_definition():
    """values()/values_at() fill large requests in chunks on several threads;
    every bit must equal the element-wise definition taken in one pass."""
    n = 2 * gen._CHUNK + 12345
    for dtype in ("f32", "bf16"):
        one = gen.normal_f32(5, 9, np.arange(777, 777 + n, dtype=np.uint64), 0.3, -0.2)
        one = one if dtype == "f32" else gen.f32_to_bf16_bits(one)
        got = gen.values(dtype, 5, 9, 777, n, 0.3, -0.2)
        assert got.dtype == one.dtype and np.array_equal(got, one)
        idx = np.random.default_rng(1).integers(0, 2 ** 40, size=(2, n // 2)).astype(np.uint64)
        at = gen.values_at(dtype, 5, 9, idx, 0.3, -0.2)
        ref = gen.normal_f32(5, 9, idx, 0.3, -0.2)
        assert at.shape == idx.shape
        assert np.array_equal(at, ref if dtype == "f32" else gen.f32_to_bf16_bits(ref))
