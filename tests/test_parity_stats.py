"""CPU checks of the parity statistic every GPU parity test relies on
(helpers.parity): max |delta logit|, raw top-1 agreement, and the count of
top-1 disagreements outside the near-tie band (oracle top-2 gap above twice
the observed max |delta|).

That last count is zero by construction: if the GPU's argmax j differs from
the oracle's i, then ref[i] - ref[j] <= (gpu[j] - ref[j]) - (gpu[i] - ref[i])
<= 2 max |delta|, and the top-2 gap is at most ref[i] - ref[j]. So the
assertions that bind in the parity tests are max |delta| <= tolerance and
the raw top-1 floors; the near-tie count is a diagnostic. The property test
below pins the bound itself."""
import numpy as np

from helpers import parity


def test_identical_logits():
    ref = np.random.Generator(np.random.PCG64(5)).normal(size=(3, 4, 50))
    assert parity(ref.copy(), ref) == (0.0, 1.0, 0)


def test_max_delta_and_agreement_counts():
    ref = np.zeros((4, 10))
    ref[:, 3] = 1.0  # clear winner 3 everywhere, gap 1.0
    gpu = ref.copy()
    gpu[0, 7] = 0.25  # a perturbation that keeps the winner
    assert parity(gpu, ref) == (0.25, 1.0, 0)
    gpu[1, 5] = 1.5  # overtakes on row 1
    maxd, agree, hard = parity(gpu, ref)
    assert (maxd, agree, hard) == (1.5, 0.75, 0)


def test_flip_inside_the_noise_band():
    ref = np.zeros((2, 6))
    ref[0, 1], ref[0, 2] = 1.00, 0.98  # gap 0.02
    ref[1, 4] = 1.0
    gpu = ref.copy()
    gpu[0, 1], gpu[0, 2] = 0.99, 0.995  # row 0 flips with max |delta| 0.015 >= gap / 2
    maxd, agree, hard = parity(gpu, ref)
    assert abs(maxd - 0.015) < 1e-12 and agree == 0.5 and hard == 0


def test_a_flip_needs_a_delta_of_half_the_gap():
    """Random logits, random perturbations at many scales: every top-1 flip
    sits where the oracle's top-2 gap is at most twice the max |delta|."""
    rng = np.random.Generator(np.random.PCG64(9))
    flips = 0
    for trial in range(300):
        ref = rng.normal(size=(8, 40))
        scale = 10.0 ** rng.uniform(-4, 0.5)
        gpu = ref + scale * rng.standard_t(3, size=ref.shape)
        maxd, agree, hard = parity(gpu, ref)
        flips += int(round((1 - agree) * ref.shape[0]))
        assert hard == 0
        srt = np.sort(ref, axis=-1)
        gap = srt[:, -1] - srt[:, -2]
        flipped = gpu.argmax(-1) != ref.argmax(-1)
        assert np.all(gap[flipped] <= 2 * maxd + 1e-12)
    assert flips > 50  # the sample does exercise flips
