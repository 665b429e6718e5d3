"""The measurement helpers on the GPU: the random-gather bandwidth and the
measured add-min peak of the integer ALU pipe that the benchmark reports its
roofline fractions against.  Both must return plausible, repeatable rates."""

import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def mpt():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_13692_gb300 import build as B

    B.build()
    from paper_2609_13692_gb300 import mpt as M

    M.load()
    return M


MAX_SM_MHZ = 2070.0  # GB300's highest SM clock


def nominal_addmin_rate():
    """SMs x 4 sub-partitions x 16 integer-ALU lanes per clock at the
    highest SM clock (an upper figure for the measured rate)."""
    props = torch.cuda.get_device_properties(0)
    return props.multi_processor_count * 64 * MAX_SM_MHZ * 1e6


def test_alu_addmin_peak_is_plausible(mpt):
    """Each add-min is one lane-operation of the 16-lane pipe: the measured
    rate must sit below the nominal SMs x 64 x clock (a compiler that folded
    the loop away would report far more) and well above a quarter of it."""
    stream = torch.cuda.current_stream().cuda_stream
    rates = [mpt.mpt_alu_addmin_peak(1 << 40, stream) for _ in range(2)]
    nominal = nominal_addmin_rate()
    for r in rates:
        assert 0.25 * nominal < r < 1.05 * nominal, (r, nominal)
    assert abs(rates[0] - rates[1]) < 0.1 * max(rates)


def test_gather_bandwidth_is_plausible(mpt):
    """Random 8-byte gathers from a 2 GiB table: between 50 GB/s and the
    copy bandwidth of the memory system."""
    gbps = mpt.mpt_gather_bandwidth(28, 1 << 26, torch.cuda.current_stream().cuda_stream)
    assert 50.0 < gbps < 8000.0, gbps
