"""The seeded input generator: published SplitMix64 values, sampling any
column set reproduces the full vector, and the distributions have the
moments the workloads ask for."""
import torch

from paper_2109_12626_gb300 import inputs as I


def _splitmix_py(state):
    M = (1 << 64) - 1
    z = state & M
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M
    return z ^ (z >> 31)


def test_splitmix64_published_first_output():
    # SplitMix64 seeded with 0: first output 0xE220A8397B1DCDAF
    z = I._mix(torch.tensor([I._s64(0x9E3779B97F4A7C15)]))
    assert int(z[0]) & ((1 << 64) - 1) == 0xE220A8397B1DCDAF


def test_words64_matches_python_ints():
    G = 0x9E3779B97F4A7C15
    for seed, rank in ((1, 0), (5, 31), (4, 1151)):
        key = _splitmix_py(seed * G + rank + 1)
        want = [_splitmix_py(key + (n + 1) * G) for n in range(64)]
        got = [v & ((1 << 64) - 1) for v in I.words64(seed, rank, torch.arange(64)).tolist()]
        assert got == want


def test_sampled_columns_equal_full_vector():
    idx = torch.tensor([0, 5, 999, 17, 3])
    for kind, kw in (("int32", dict(lo=-1000, hi=1000)),
                     ("float32", dict(sigma=1e-3)), ("mat2x2u32", {})):
        full = I.rank_values(kind, 9, 4, 1000, **kw)
        part = I.rank_values(kind, 9, 4, idx, **kw)
        assert torch.equal(full[idx], part)


def test_distributions():
    u = I.uniform_int32(3, 0, 200000, -(1 << 20), 1 << 20)
    assert int(u.min()) >= -(1 << 20) and int(u.max()) <= 1 << 20
    assert abs(float(u.double().mean())) < 0.02 * (1 << 20)
    v = I.normal_f32(4, 0, 200000)
    assert abs(float(v.mean())) < 0.01 and abs(float(v.std()) - 1) < 0.01
    assert float(v.abs().max()) <= 6.0
    w = I.normal_f32(5, 0, 100000, sigma=1e-3)
    assert abs(float(w.std()) - 1e-3) < 2e-5
    m = I.words_u32(2, 0, 50000, 4).view(torch.int32).to(torch.int64) & 0xFFFFFFFF
    assert abs(float(m.double().mean()) / 2**32 - 0.5) < 0.01
    assert not torch.equal(I.normal_f32(4, 0, 64), I.normal_f32(4, 1, 64))
