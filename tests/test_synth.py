"""The seeded input generator against its published definition and basic statistics."""
import json
import os

import numpy as np

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
M64 = (1 << 64) - 1


def _splitmix64(state):
    # SplitMix64 as published: state += gamma; output = finalizer(state).
    while True:
        state = (state + 0x9E3779B97F4A7C15) & M64
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
        yield z ^ (z >> 31)


def test_splitmix_published_vector():
    g = json.load(open(os.path.join(GOLDEN, "splitmix64.json")))
    it = _splitmix64(g["state"])
    assert [next(it) for _ in range(5)] == g["outputs"]


def test_raw_draw_is_counter_based_splitmix():
    # The stream key is itself a SplitMix64 finalizer mix; draw i of a stream is
    # output i of SplitMix64 started from that key.
    def fin(z):
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
        return z ^ (z >> 31)
    seed, stream = 7, 3
    key = fin((seed * 0x9E3779B97F4A7C15 + 0x9E3779B97F4A7C15) & M64) ^ fin(((stream + 1) * 0xD1B54A32D192ED03) & M64)
    it = _splitmix64(key)
    assert [next(it) for _ in range(6)] == [synth.raw_draw(seed, stream, i) for i in range(6)]


def test_thread_count_and_offset_invariance():
    a = synth.normal(5, 9, (300000,), "f32", nthreads=1)
    b = synth.normal(5, 9, (300000,), "f32", nthreads=7)
    assert np.array_equal(a, b)
    c = synth.normal(5, 9, (1000,), "f32", offset=123456)
    assert np.array_equal(c, a[123456:124456])
    ia = synth.uniform_int(1, 0, (200000,), 0, 151936, nthreads=1)
    ib = synth.uniform_int(1, 0, (200000,), 0, 151936, nthreads=5)
    assert np.array_equal(ia, ib)


def test_normal_statistics():
    x = synth.normal(0, 1, (1 << 20,), "f32").astype(np.float64)
    assert abs(x.mean()) < 5e-3 and abs(x.std() - 1) < 5e-3
    # fourth moment of a normal is 3
    assert abs(np.mean(x ** 4) - 3) < 0.05


def test_bf16_is_rne_of_f32():
    f = synth.normal(4, 2, (100000,), "f32", sigma=0.02)
    h = synth.normal(4, 2, (100000,), "bf16", sigma=0.02)
    u = f.view(np.uint32).astype(np.uint64)
    rne = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    assert np.array_equal(rne, h)


def test_uniform_int_range():
    t = synth.uniform_int(1, 0, (500000,), 0, 4096)
    assert t.min() >= 0 and t.max() < 4096
    counts = np.bincount(t, minlength=4096)
    assert counts.min() > 50 and counts.max() < 200


def test_tensor_list_shapes():
    s = synth.shape("q8b")
    tl = synth.tensor_list(s)
    assert len(tl) == 3 + 11 * 36
    params = sum(int(np.prod(t[1])) for t in tl)
    # Qwen3-8B with a separate lm_head: 8.19 G parameters
    assert 8.18e9 < params < 8.20e9
    streams = [t[3] for t in tl]
    assert len(set(streams)) == len(streams)


def test_row_range_generation_matches_full():
    s = synth.shape("tiny_fp32")
    full = synth.gen_tensor(s, "layers.1.wd")
    part = synth.gen_tensor(s, "layers.1.wd", rows=(10, 20))
    assert np.array_equal(full[10:20], part)
    g = synth.gen_tensor(s, "final_norm")
    assert abs(g.mean() - 1) < 0.01 and 0.01 < g.std() < 0.03
