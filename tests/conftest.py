import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the CUDA path through the C-ABI)")
    config.addinivalue_line("markers", "slow: full-size parity case (minutes)")


def load_golden_sha256():
    """Parse tests/golden/fips180_2_sha256_examples.txt -> [(message bytes, digest bytes)]."""
    out = []
    path = os.path.join(ROOT, "tests", "golden", "fips180_2_sha256_examples.txt")
    with open(path) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            spec, hexd = line.split()
            if "*" in spec:
                ch, count = spec.split("*")
                msg = ch.encode() * int(count)
            else:
                msg = spec.encode()
            out.append((msg, bytes.fromhex(hexd)))
    return out


@pytest.fixture(scope="session")
def golden_sha256():
    return load_golden_sha256()


def load_golden_base64():
    """Parse tests/golden/rfc4648_base64_vectors.txt -> [(input bytes, encoding str)]."""
    out = []
    path = os.path.join(ROOT, "tests", "golden", "rfc4648_base64_vectors.txt")
    with open(path) as f:
        for line in f:
            line = line.rstrip("\n")
            if not line or line.startswith("#"):
                continue
            a, b = line.split("\t")
            out.append((b"" if a == "<empty>" else a.encode(), "" if b == "<empty>" else b))
    return out
