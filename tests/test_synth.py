"""The synthetic rollout recipe (input generation only): GRPO group-normalised
advantages, response-length masks and the DAPO dynamic-sampling filter, on the
workload shapes.  These pin the inputs the parity tests and the bench use."""

import dataclasses

import numpy as np
import pytest

from paper_2609_22870_gb300 import synth


def _groups(w, x):
    return np.asarray(x).reshape(w.prompts, w.group, w.resp_len)


@pytest.mark.parametrize("name", ["grpo_8b", "dapo_32b", "long_8b"])
def test_advantages_are_group_normalised(name):
    w = synth.WORKLOADS[name]
    adv, _ = synth.rollout(w)
    A = _groups(w, adv.numpy())[:, :, 0].astype(np.float64)  # one value per response
    assert np.all(_groups(w, adv.numpy()) == A[:, :, None])  # broadcast over the response
    for a in A:
        if np.all(a == 0):  # all-equal rewards
            continue
        assert abs(a.mean()) < 1e-5
        assert abs(a.std(ddof=1) - 1.0) < 1e-4  # (R - mean) / (std + 1e-6), unbiased std


def test_length_mask_is_a_prefix_of_each_response():
    w = synth.WORKLOADS["grpo_8b"]
    _, mask = synth.rollout(w)
    m = _groups(w, mask.numpy()).reshape(-1, w.resp_len)
    lengths = m.sum(1)
    assert lengths.min() >= w.length_mask[0] and lengths.max() <= w.length_mask[1]
    for row, n in zip(m, lengths):
        assert np.all(row[:n] == 1) and np.all(row[n:] == 0)


def test_dapo_filter_masks_exactly_the_all_equal_groups():
    w = dataclasses.replace(synth.WORKLOADS["dapo_32b"], T=4 * 16 * 64, resp_len=64)
    adv, mask = synth.rollout(w, force_equal_prompt=2)
    A = _groups(w, adv.numpy())[:, :, 0]
    M = _groups(w, mask.numpy())
    equal = np.all(A == A[:, :1], axis=1)
    assert equal[2]  # the forced group
    for p in range(w.prompts):
        assert np.all(M[p] == (0 if equal[p] else 1))
        if equal[p]:
            assert np.all(A[p] == 0)
    # without the filter the forced group stays valid (A = 0 tokens belong to neither sign)
    w2 = dataclasses.replace(w, filter_equal_groups=False)
    adv2, mask2 = synth.rollout(w2, force_equal_prompt=2)
    assert np.all(_groups(w2, mask2.numpy())[2] == 1) and np.all(_groups(w2, adv2.numpy())[2] == 0)
