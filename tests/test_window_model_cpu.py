"""The prefix-window call's launch-time choice between the packed grouped-query kernel and the
square kernel (host arithmetic, no GPU): the shapes the packed kernel runs, the split of the keys
it takes, and the choice on the windows measured on GB300, given that GPU's resident-cluster
counts for the packed kernel (cudaOccupancyMaxActiveClusters at its 205.6 KB of shared memory:
152, 76, 46, 36, 28, 23, 15, 15 clusters of 1 .. 8 CTAs; 152 SMs)."""
import pytest

from paper_2602_06161_gb300 import CoverError, api

GB300 = dict(n_sm=152, max_clusters=[152, 76, 46, 36, 28, 23, 15, 15])


def _model(B, Hq, Hkv, Lk, Lq, q0=None, **gpu):
    gpu = gpu or GB300
    return api.cover_debug_window_model(B, Hq, Hkv, Lq, Lk, Lk - Lq if q0 is None else q0, gpu["n_sm"],
                                        gpu["max_clusters"])


@pytest.mark.parametrize("B,Hq,Hkv,Lk,Lq,packed", [
    # the windows measured on GB300 (calls back to back): the faster kernel of each
    (1, 28, 4, 1024, 16, True),      # 8.3 against 12.1 us
    (1, 28, 4, 1024, 32, True),      # 8.7 against 12.1 us (Dream block)
    (1, 28, 4, 1024, 64, False),     # 14.9 against 12.1 us: 16 clusters of 8, two waves
    (1, 28, 4, 1024, 128, False),    # 17.4 against 12.4 us
    (4, 28, 4, 1024, 32, False),     # 24.2 against 13.4 us
    (1, 28, 4, 4096, 32, True),      # 13.0 against 32.9 us
    (1, 32, 8, 8192, 32, True),      # 18.8 against 60.6 us
    (1, 32, 8, 8192, 64, True),      # 36.5 against 60.7 us
    (8, 32, 8, 2048, 64, False),     # 90.1 against 39.7 us
    (2, 16, 2, 2048, 32, True),      # 10.2 against 19.1 us
])
def test_choice_on_the_measured_windows(B, Hq, Hkv, Lk, Lq, packed):
    c = _model(B, Hq, Hkv, Lk, Lq)
    assert c["supported"] and c["resident"]
    assert c["packed"] == packed, c


def test_split_of_the_keys():
    # T = ceil(nkv / 8) KV tiles per CTA, nsplit = ceil(nkv / T) CTAs per cluster
    for Lk, T, nsplit in ((90, 1, 1), (129, 1, 2), (1024, 1, 8), (1100, 2, 5), (2048, 2, 8), (4096, 4, 8),
                          (8192, 8, 8), (8100, 8, 8), (1025, 2, 5)):
        c = _model(1, 8, 2, Lk, 16)
        assert (c["T"], c["nsplit"]) == (T, nsplit), (Lk, c)
    # Q tiles per KV head: ceil(G Lq / 128)
    for Hq, Hkv, Lq, n_qt in ((28, 4, 32, 2), (28, 4, 128, 7), (8, 2, 32, 1), (9, 3, 37, 1), (4, 2, 128, 2)):
        assert _model(1, Hq, Hkv, 1024, Lq)["n_qt"] == n_qt


def test_shapes_the_packed_kernel_does_not_run():
    assert not _model(1, 32, 32, 1024, 32)["supported"]          # G = 1: nothing to pack
    assert not _model(1, 28, 4, 1024, 1024, q0=0)["supported"]   # the square call
    assert not _model(1, 8, 2, 1024, 257)["supported"]           # more than 256 window rows
    assert not _model(1, 28, 4, 1024, 160)["supported"]          # 1120 packed rows > 1024
    assert not _model(1, 8, 2, 8193, 32)["supported"]            # more than 64 KV tiles
    assert _model(1, 8, 2, 8192, 128)["supported"]               # the limits themselves
    c = _model(1, 32, 32, 1024, 32)
    assert not c["packed"] and c["T"] == 0 and c["packed_us"] == 0.0


def test_a_cluster_that_cannot_be_resident_leaves_the_square_kernel():
    gpu = dict(n_sm=152, max_clusters=[152, 76, 46, 36, 28, 23, 15, 0])
    c = _model(1, 28, 4, 1024, 32, **gpu)
    assert c["supported"] and not c["resident"] and not c["packed"]


def test_waves_of_clusters_in_the_prediction():
    # the packed prediction grows by whole waves of resident clusters; the square one by rounds
    one = _model(1, 28, 4, 1024, 32)        # 8 clusters of 8: one wave
    two = _model(2, 28, 4, 1024, 32)        # 16 clusters of 8: two waves
    assert two["packed_us"] == pytest.approx(2 * one["packed_us"])
    assert one["square_us"] == pytest.approx(two["square_us"])   # 28 and 56 units: one round each


def test_invalid_arguments():
    with pytest.raises(CoverError):
        api.cover_debug_window_model(1, 28, 5, 32, 1024, 992, 152, GB300["max_clusters"])   # Hq % Hkv
    with pytest.raises(CoverError):
        api.cover_debug_window_model(1, 28, 4, 32, 1024, 1000, 152, GB300["max_clusters"])  # q0 + Lq > Lk
    with pytest.raises(CoverError):
        api.cover_debug_window_model(1, 28, 4, 32, 1024, 992, 0, GB300["max_clusters"])     # no SMs
