"""The work counts behind bench.py's rooflines, on the CPU.

SHA-256 pads a message of L bytes to floor((L + 8) / 64) + 1 blocks of 64
bytes (FIPS 180-4 5.1.1: a 0x80 byte, zeros, and the 64-bit length), so a
chunk of C int32 tokens costs floor((4C + 8) / 64) + 1 compressions and a
chain step (k_{i-1} || d || c_i, 96 bytes) costs 2.  The per-configuration
totals are those of the workload table of the measurement plan: multi-adapter
278,528 digest and 32,768 chain compressions, small-block 4,194,304 and
4,194,304, long context 557,056 and 65,536, each sweep 2,228,224 and 262,144,
tiny 272 and 32.
"""
import pytest

import bench


def blocks(L: int) -> int:
    return (L + 8) // 64 + 1


@pytest.mark.parametrize("C", list(range(1, 300)) + [1000, 4096, 250000])
def test_compressions_per_chunk_follow_the_padding_rule(C):
    dig, chain = bench.compressions(1, C)
    assert dig == blocks(4 * C)
    assert chain == 2 == blocks(96)


@pytest.mark.parametrize("name, R, T, C, dig, chain", [
    ("tiny", 8, 512, 256, 272, 32),
    ("multi_adapter", 1024, 4096, 256, 278_528, 32_768),
    ("small_block", 16384, 2048, 16, 4_194_304, 4_194_304),
    ("long_context", 64, 131072, 256, 557_056, 65_536),
    ("provenance_sweep", 4096, 8192, 256, 2_228_224, 262_144),
])
def test_per_configuration_compressions(name, R, T, C, dig, chain):
    assert bench.compressions(R * (T // C), C) == (dig, chain)


def test_critical_path_of_the_multi_adapter_batch():
    """17 compressions for the first chunk digest, then 2 per chunk of a 16-chunk request: 49 in series,
    each at least 64 rounds x 10 logic/shift instructions x 2 cycles = 1280 cycles at the max SM clock."""
    import numpy as np

    class Batch:
        R = 3
        tok_off = np.array([0, 4096, 8192, 12288], np.int64)

    class Wl:
        chunk_tokens = 256
        batch = Batch()

    cp = bench.critical_path(Wl(), 74e-6, {"sm_max_mhz": 2070.0})
    assert cp["serial_compressions"] == 49
    assert abs(cp["compression_floor_us"] - 1280 / 2070) < 1e-12
    assert abs(cp["bound_us"] - 49 * 1280 / 2070) < 1e-9
    assert abs(cp["frac"] - cp["bound_us"] / 74.0) < 1e-12


def test_ops_per_compression():
    # 64 rounds x (6 rotations + 4 three-input logic + 4 adds) + 48 schedule words x (6 + 2 + 2) + 8 feed-forward
    assert bench.SHA_OPS_PER_COMPRESSION == 64 * 14 + 48 * 10 + 8 == 1384


def test_auto_steps_give_a_timed_region_of_at_least_the_minimum():
    import bench
    for it in (0.2e-3, 0.9e-3, 1.4e-3, 7e-3):
        k = bench.auto_steps(it)
        assert k * it >= bench.MIN_TIMED_S or k == 4000
        assert (k - 1) * it < bench.MIN_TIMED_S or k == 20
    assert bench.auto_steps(10.0) == 20 and bench.auto_steps(1e-9) == 4000 and bench.auto_steps(0) == 20
