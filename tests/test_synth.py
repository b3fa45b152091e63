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


def test_compiled_host_generator_equals_the_numpy_definition():
    """gen_host.c (the fast host fill) gives every bit the numpy definition
    gives, for consecutive runs and scattered indices, both storage dtypes."""
    L = gen._host_lib()
    assert L is not None, "gen_host.c did not build"
    rng = np.random.default_rng(7)
    for dtype in ("f32", "bf16"):
        for seed, stream, start, n, std, mean in [(0, 30, 0, 100003, 1.0, 0.0),
                                                  (3, 4, 2 ** 33 + 5, 70001, 0.1, 1.0),
                                                  (1, 40, 12345, 1, 8.0, 0.0),
                                                  (2, 10, 2 ** 40, 300000, 0.0625, -0.5)]:
            a = gen.values(dtype, seed, stream, start, n, std, mean)
            b = gen.values_np(dtype, seed, stream, start, n, std, mean)
            assert a.dtype == b.dtype and np.array_equal(a, b), (dtype, seed, stream)
            idx = rng.integers(0, 2 ** 50, size=(3, 1001)).astype(np.uint64)
            a = gen.values_at(dtype, seed, stream, idx, std, mean)
            b = gen.values_at_np(dtype, seed, stream, idx, std, mean)
            assert a.shape == idx.shape and np.array_equal(a, b)


def test_runs_gather_equals_consecutive_values():
    starts = np.array([5, 2 ** 35 + 3, 999, 5], dtype=np.uint64)
    for dtype in ("f32", "bf16"):
        got = gen.values_runs(dtype, 4, 31, starts, 4097, 0.5, 0.25)
        for r, s0 in enumerate(starts):
            assert np.array_equal(got[r], gen.values_np(dtype, 4, 31, int(s0), 4097, 0.5, 0.25))
