"""The seeded input generator: Philox known answers, determinism, recipes."""
import hashlib

import numpy as np
import pytest

from paper_2608_26004_gb300 import synth


def test_philox4x32_10_known_answers():
    # Known-answer vectors of Philox4x32-10 published with the algorithm.
    assert synth.philox4x32_10((0, 0, 0, 0), (0, 0)) == (
        0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)
    assert synth.philox4x32_10((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2) == (
        0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)
    assert synth.philox4x32_10((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344),
                               (0xA4093822, 0x299F31D0)) == (
        0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1)


def _digest(batch):
    h = hashlib.sha256()
    for x in (batch.logits_full, batch.logits_comp, batch.logits_ver, batch.draft_tokens,
              batch.draft_probs, batch.uniforms):
        h.update(np.ascontiguousarray(x).tobytes())
    return h.hexdigest()


def test_generation_is_deterministic_and_thread_count_free():
    a = synth.make_config(0, nthreads=1)
    b = synth.make_config(0, nthreads=5)
    assert _digest(a) == _digest(b)


def test_sample_of_batch_equals_slice_of_full_batch():
    full = synth.make_config(1, nb=4)
    part = synth.make_config(1, b0=2, nb=2)
    for name in ("logits_full", "logits_comp", "logits_ver", "draft_tokens", "draft_probs",
                 "uniforms"):
        assert np.array_equal(getattr(full, name)[2:4], getattr(part, name)), name


def test_recipe_gaussian_spike_and_perturbation_fraction():
    b = synth.make_config(0)
    v = b.logits_ver.astype(np.float64)
    f = b.logits_full.astype(np.float64)
    c = b.logits_comp.astype(np.float64)
    # one +8 spike per row on top of N(0, 2^2)
    assert np.all(v.max(axis=2) > 6.0)
    assert np.std(np.sort(v, axis=2)[..., :-1]) == pytest.approx(2.0, rel=0.02)
    assert np.std(f - v) == pytest.approx(0.5, rel=0.02)
    moved = c != f
    assert moved.mean() == pytest.approx(0.05, abs=0.003)
    assert np.std((c - f)[moved]) == pytest.approx(3.0, rel=0.05)
    assert np.all((b.uniforms >= 0) & (b.uniforms < 1))
    assert np.all((b.draft_tokens >= 0) & (b.draft_tokens < b.V))


def test_recipe_identical_lower_half_for_large_batch_config():
    b = synth.make_config(3, b0=126, nb=4)        # elements 126..129 of B = 256
    assert np.array_equal(b.logits_full[:2], b.logits_comp[:2])
    moved = (b.logits_full[2:] != b.logits_comp[2:]).mean()
    assert moved == pytest.approx(0.20, abs=0.01)


def test_recipe_zipf_profile_is_permuted_sorted_ranks():
    b = synth.make_config(2, nb=1)
    v = synth.bf16_bits_to_f32(b.logits_ver[0, 0]).astype(np.float64)
    V = v.size
    srt = np.sort(v)[::-1]
    ranks = np.arange(1, V + 1)
    # sorted values follow -1.1 ln(rank) up to the N(0, 0.3^2) noise
    assert np.median(np.abs(srt - (-1.1 * np.log(ranks)))) < 0.5
    assert np.argmax(v) != 0 or np.argmax(synth.bf16_bits_to_f32(b.logits_ver[0, 1])) != 0


def test_draft_probs_are_drafter_probabilities_of_drafts():
    b = synth.make_config(0)
    a = b.logits_full[0].astype(np.float64)
    for k in range(b.K):
        z = a[k] - a[k].max()
        p = np.exp(z) / np.exp(z).sum()
        assert b.draft_probs[0, k] == pytest.approx(p[b.draft_tokens[0, k]], rel=1e-6)


def test_xvocab_inputs_embed_the_shared_set():
    # the recipe generated over the S shared tokens, scattered through a map
    # whose two sides are injective and in range
    w = synth.CONFIGS[1]
    x = synth.make_xvocab(w.recipe, w.seed, 2, 3, 200, 300, 250, synth.BF16)
    inner = synth.generate(w.recipe, w.seed, 2, 3, 200, synth.BF16)
    assert np.unique(x.map_d).size == 200 and np.all(np.diff(x.map_d) > 0)
    assert np.unique(x.map_v).size == 200 and 0 <= x.map_v.min() and x.map_v.max() < 250
    assert x.map_d.max() < 300
    assert np.array_equal(x.logits_full[..., x.map_d], inner.logits_full)
    assert np.array_equal(x.logits_comp[..., x.map_d], inner.logits_comp)
    assert np.array_equal(x.logits_ver[..., x.map_v], inner.logits_ver)
    assert np.array_equal(x.draft_tokens, inner.draft_tokens)
    assert np.array_equal(x.draft_probs, inner.draft_probs)
    # reproducible from the seed
    y = synth.make_xvocab(w.recipe, w.seed, 2, 3, 200, 300, 250, synth.BF16)
    assert np.array_equal(x.logits_ver, y.logits_ver) and np.array_equal(x.map_v, y.map_v)
    # bf16 rounding of the unpaired fill is round-to-nearest-even
    bits = synth._f32_to_bf16_bits(np.array([1.0, 1 + 2**-8, 1 + 3 * 2**-8, -2.5], np.float32))
    assert list(bits) == [0x3F80, 0x3F80, 0x3F82, 0xC020]
