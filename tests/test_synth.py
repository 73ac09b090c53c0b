"""The seeded input generator: determinism, slicing, exact counts, shapes
of the distributions the workloads ask for (CPU only)."""
import numpy as np

from paper_2609_35440_gb300 import synth, workloads


def test_deterministic_and_sliceable():
    wl = workloads.SMOKE
    a = synth.gen_hidden(wl, 1)
    b = synth.gen_hidden(wl, 1)
    assert a.dtype == np.uint16 and np.array_equal(a, b)
    part = synth.gen_hidden(wl, 1, row0=37, rows=11)
    assert np.array_equal(part, a[37:48])
    assert not np.array_equal(synth.gen_hidden(wl, 0), a)


def test_normal_moments_and_bf16():
    x = synth.normal(5, 1, 0, 200000)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1) < 0.01
    bits = synth.to_bf16_bits(np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5]))
    assert list(synth.bf16_bits_to_f32(bits)) == [1.0, 1.0, 1.0 + 2 ** -6, -2.5]


def test_masks_heavy_rows_and_zipf():
    wl = workloads.vocab_sweep(32000).with_(N=1000, d=256)
    y = synth.gen_targets(wl)
    assert np.all((y == -100).sum(axis=1) == 50)
    W = synth.bf16_bits_to_f32(synth.gen_W(wl)).astype(np.float64)
    rms = np.sqrt(np.mean(W ** 2, axis=1))
    assert int((rms > 0.1).sum()) == 320          # exactly 1% of rows x20
    z = workloads.W1P3B.with_(N=20000, V=1000, mask_frac=0.0)
    t = synth.gen_targets(z)[0]
    freq = np.bincount(t, minlength=1000) / len(t)
    w = np.arange(1, 1001, dtype=float) ** -1.1
    w /= w.sum()
    assert abs(freq[0] - w[0]) < 0.01 and abs(freq[9] - w[9]) < 0.005
    assert t.min() >= 0 and t.max() < 1000


def test_row_scale_range():
    wl = workloads.W1P3B.with_(N=64, d=512)
    h = synth.bf16_bits_to_f32(synth.gen_hidden(wl, 0)).astype(np.float64)
    rms = np.sqrt(np.mean(h ** 2, axis=1))
    assert rms.min() > 0.4 and rms.max() < 9.0 and rms.max() / rms.min() > 4
