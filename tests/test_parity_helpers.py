"""The parity comparator of the GPU tests, checked on the CPU with planted disagreements.

The edge-value tests rely on tests.gpu_helpers.assert_close_special to compare NaN, infinities,
out-of-range and subnormal results with the fp64 oracle; a comparator that accepts a wrong
class or sign would let a kernel bug through, so each rule is exercised here both ways."""
import numpy as np
import pytest

from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import FINITE_MAX, assert_close_special, subnormal_floor

F32, BF16 = bc.DTYPE_F32, bc.DTYPE_BF16
inf, nan = np.inf, np.nan


def f32(*v):
    return np.array(v, dtype=np.float32)


def test_matching_classes_pass():
    ref = np.array([1.0, nan, inf, -inf, 9.9e38, -9.9e38, 0.0])
    bound = np.array([1.0, nan, inf, inf, 9.9e38, 9.9e38, 0.0])
    assert_close_special(f32(1.0, nan, inf, -inf, inf, -inf, -0.0), ref, bound, F32)
    bits = synth.f32_to_bf16_bits(f32(1.0, nan, inf, -inf, inf, -inf, 0.0))
    assert_close_special(bits, ref, bound, BF16)


@pytest.mark.parametrize("gpu,ref,bound", [
    (f32(inf), [3.0e38], [3.0e38]),          # overflow where the result is representable
    (f32(1.0), [nan], [nan]),                # NaN lost
    (f32(nan), [inf], [inf]),                # infinity turned into NaN
    (f32(-inf), [inf], [inf]),               # wrong sign of an infinity
    (f32(-inf), [9.9e38], [9.9e38]),         # out of range: the infinity of the wrong sign
    (f32(3.0e38), [9.9e38], [9.9e38]),       # out of range but finite on the GPU
    (f32(1.001), [1.0], [1.0]),              # plain error beyond 1e-5
])
def test_disagreements_fail(gpu, ref, bound):
    with pytest.raises(AssertionError):
        assert_close_special(gpu, np.array(ref), np.array(bound), F32)


def test_range_edge_uses_the_output_type():
    # 3.3e38 is finite in fp32 but beyond the largest bf16 value: a bf16 infinity is right
    # there only if the oracle's value exceeds the bf16 maximum by more than the tolerance
    ref = np.array([3.39e38])
    assert FINITE_MAX[BF16] < ref[0] < FINITE_MAX[F32]
    assert_close_special(f32(3.39e38), ref, ref, F32)
    assert_close_special(np.array([0x7F7F], dtype=np.uint16), ref, ref, BF16)   # bf16 max
    with pytest.raises(AssertionError):
        assert_close_special(f32(inf), ref, ref, F32)


def test_subnormal_floor():
    # two subnormal fp32 values one spacing (2^-149) apart differ by far more than 1e-5 of
    # their size: only the absolute floor admits them, and it is a handful of spacings
    tiny = 2.0 ** -140
    ref = np.array([tiny])
    gpu = f32(tiny + 2.0 ** -149)
    with pytest.raises(AssertionError):
        assert_close_special(gpu, ref, ref, F32)
    fl = subnormal_floor(3, 7.0, F32)
    assert 2.0 ** -149 < fl < 64 * 2.0 ** -149
    assert_close_special(gpu, ref, ref, F32, fl)
    assert subnormal_floor(3, 7.0, BF16) - fl == 2.0 ** -134
