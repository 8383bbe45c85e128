"""The seeded synthetic streams that stand in for the paper's benchmark
videos: the counter-based generator against SplitMix64's published outputs,
determinism and slicing, and the structure each recipe promises (scene
lengths, injected events, push sizes, noise level). CPU only."""
import numpy as np

import synth


def test_splitmix64_published_outputs():
    """synth.u64(key, i) is the i-th output of SplitMix64 (Steele, Lea and
    Flood, 2014) seeded with key; the first outputs for seed 0 are the
    generator's published test values."""
    assert synth.u64(0, 0) == 0xE220A8397B1DCDAF
    assert synth.u64(0, 1) == 0x6E789E6AA1B965F4
    assert synth.u64(0, 2) == 0x06C45D188009454F


def test_generation_is_seeded_and_sliceable():
    spec = synth.medium(seed=7).with_(width=40, height=24, frames=50)
    a = synth.generate(spec)
    assert a.shape == (50, 24, 40, 3) and a.dtype == np.uint8
    assert np.array_equal(a, synth.generate(spec, nthreads=1)), "the thread count changes nothing"
    assert np.array_equal(a[17:33], synth.generate(spec, 17, 33)), "any slice is generated on its own"
    assert not np.array_equal(a, synth.generate(spec.with_(seed=8))), "the seed matters"


def test_stream_shapes():
    assert (synth.tiny().frames, synth.tiny().width, synth.tiny().height) == (64, 224, 224)
    assert (synth.medium().frames, synth.medium().width, synth.medium().height) == (600, 448, 448)
    assert (synth.hd1080().frames, synth.hd1080().width, synth.hd1080().height) == (3600, 1920, 1080)
    assert synth.hd1080().total_bytes == 22_394_880_000
    serving = [synth.serving_stream(s) for s in range(synth.SERVING_STREAMS)]
    assert len({s.seed for s in serving}) == 32 and all((s.frames, s.width, s.height) == (1800, 640, 360)
                                                        for s in serving)
    r = synth.rare_event()
    assert (r.frames, r.width, r.height, r.n_events) == (3600, 1280, 720, 40)


def test_scene_structure():
    assert synth.scene_starts(synth.tiny()).tolist() == [0, 16, 32, 48]  # 4 scenes of 16 frames
    for spec, mean in ((synth.medium(), 20), (synth.hd1080(), 150), (synth.rare_event(), 20)):
        starts = synth.scene_starts(spec)
        assert starts[0] == 0 and np.all(np.diff(starts) >= 1) and starts[-1] < spec.frames
        lengths = np.diff(np.append(starts, spec.frames))
        # geometric scene lengths: the sample mean is within a loose band around the recipe's mean
        assert 0.5 * mean <= lengths.mean() <= 2.0 * mean, (spec, lengths.mean())


def test_rare_event_stream_has_short_events():
    m = synth.event_mask(synth.rare_event())
    edges = np.flatnonzero(np.diff(np.concatenate([[0], m, [0]])))
    runs = edges[1::2] - edges[::2]
    # 40 events of 1-3 frames at random positions: adjacent or overlapping ones merge into one run
    assert 30 <= runs.size <= 40 and 40 <= m.sum() <= 120 and runs.min() >= 1
    assert m.sum() <= 3 * 40


def test_serving_push_sizes_are_uniform_1_to_8():
    sizes = synth.push_sizes(synth.SEED_BASE + 4, 0, 16000)
    assert sizes.min() == 1 and sizes.max() == 8
    counts = np.bincount(sizes, minlength=9)[1:]
    assert np.all(np.abs(counts - 2000) < 200), counts  # about 4.5 sigma of a fair 1/8 draw


def test_noise_level_within_a_scene():
    """Consecutive frames of one tiny scene differ only by the sigma = 4 noise
    (apart from clamping): their difference has a standard deviation near
    4 sqrt(2)."""
    a = synth.generate(synth.tiny(), 0, 2).astype(np.int32)
    d = (a[1] - a[0]).ravel()
    assert 4.0 <= d.std() <= 7.5 and abs(d.mean()) < 0.5
