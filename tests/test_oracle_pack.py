"""Pins for the oracle's initialisation, hard projection and packing:
  * its fp32 -> fp16 converter agrees with numpy's IEEE cast (library routine);
  * unpack(pack(c)) = c, and hand-derived bit patterns for the stream layout;
  * storage accounting matches Table 1 (2.13, 3.13, 1.71 bit/param at group 128);
  * round-to-nearest codes land on exact grid points; absmax scale maps the largest
    weight onto the outermost level; projection picks the largest logit.
"""
import numpy as np
import pytest

from oracle import gsq_oracle as O


def test_fp16_converter_matches_ieee_cast():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        (rng.standard_normal(200000) * 10.0 ** rng.integers(-9, 6, 200000)).astype(np.float32),
        np.array([0.0, -0.0, 65504, 65519.99, 65520, -65520, 1e9, np.inf, -np.inf,
                  2 ** -24, 2 ** -25, 3 * 2 ** -26, 2 ** -14, 2 ** -14 - 2 ** -25,
                  1 + 2 ** -11, 1 + 3 * 2 ** -11, 6e-8, 1e-30], dtype=np.float32),
    ]).astype(np.float32)
    ours = O.f32_to_f16_bits(x)
    with np.errstate(over="ignore"):
        ref = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(ours, ref)
    assert O.f32_to_f16_bits(np.float32([np.nan]))[0] & 0x7C00 == 0x7C00
    fin = np.isfinite(x) & (np.abs(x) < 65520)
    back = O.f16_bits_to_f32(ref[fin])
    assert np.array_equal(back, x[fin].astype(np.float16).astype(np.float32))


def test_pack_stream_hand_patterns():
    # 2-bit: codes 0,1,2,3 repeated -> every byte 0b11_10_01_00 = 0xE4
    codes = np.tile(np.arange(4, dtype=np.uint8), 8)
    buf = O.pack_group(codes, np.float32([1.0, 1.0]), K=4)
    assert buf[:8] == bytes([0xE4] * 8)
    assert buf[16:20] == bytes([0x00, 0x3C, 0x00, 0x3C])      # fp16(1.0) = 0x3C00, LE
    # 3-bit: codes 0..7 repeated; in octal, the 96-bit word reads 76543210 x 4
    codes = np.tile(np.arange(8, dtype=np.uint8), 4)
    buf = O.pack_group(codes, np.float32([1.0]), K=8)
    assert buf[:12] == int("76543210" * 4, 8).to_bytes(12, "little")


@pytest.mark.parametrize("K", [3, 4, 5, 8])
def test_pack_roundtrip_group(K):
    rng = np.random.default_rng(K)
    n, G = 4096 + 64, 64
    codes = rng.integers(0, K, n).astype(np.uint8)
    scales = (rng.standard_normal(n // G) * 0.01).astype(np.float32)
    buf = O.pack_group(codes, scales, K)
    assert len(buf) == O.code_section_bytes(n, K) + 2 * (n // G)
    c2, s2 = O.unpack_group(buf, n, K, n // G)
    assert np.array_equal(c2, codes)
    assert np.array_equal(s2, O.f32_to_f16_bits(scales))


def test_pack_roundtrip_kquant2():
    rng = np.random.default_rng(11)
    n = 256 * 12
    codes = rng.integers(0, 8, n).astype(np.uint8)
    d = np.float32(rng.random(n // 256) * 1e-3)
    d = O.f16_bits_to_f32(O.f32_to_f16_bits(d))
    sc = rng.integers(-32, 32, n // 16).astype(np.int32)
    buf = O.pack_kquant2(codes, d, sc)
    assert len(buf) == 110 * (n // 256)
    c2, d2, sc2 = O.unpack_kquant2(buf, n)
    assert np.array_equal(c2, codes) and np.array_equal(d2, d) and np.array_equal(sc2.reshape(-1), sc)
    # 110 bytes per 256 weights = 3.4375 bit/weight
    assert 110 * 8 / 256 == 3.4375


def test_storage_accounting_matches_table1():
    # Table 1 prints two decimals (2.125 -> 2.13, half rounded up)
    assert abs(O.bits_per_param(4, 128) - 2.13) <= 0.005
    assert abs(O.bits_per_param(8, 128) - 3.13) <= 0.005
    assert abs(O.bits_per_param(3, 128) - 1.71) <= 0.005
    # the packed group format at b bits + fp16 per group of 128 realises b + 0.125
    n, G = 128 * 1024, 128
    for K, b in ((4, 2), (8, 3)):
        size = O.code_section_bytes(n, K) + 2 * (n // G)
        assert size * 8 / n == b + 16 / G


def test_rtn_codes_and_absmax_scale():
    grid = np.array([-1.5, -0.5, 0.5, 1.5])
    s = np.float32(0.0125)
    codes = np.array([0, 3, 1, 2, 2, 1, 3, 0] * 16, dtype=np.uint8)
    W = (s * grid[codes].astype(np.float32)).astype(np.float32).reshape(1, -1)
    sc = O.init_group_scales(W, 128, grid)
    assert sc[0, 0] == np.float32(np.abs(W).max() / np.float32(1.5))
    got = O.rtn_codes(W, np.repeat(sc, 128, 1), grid)
    assert np.array_equal(got.reshape(-1), codes)
    # ties go to the lower level: W/s exactly between -0.5 and 0.5
    assert O.rtn_codes(np.float32([[0.0]]), np.float32([[1.0]]), grid)[0, 0] == 1
    # out-of-range clamps to the end levels
    assert O.rtn_codes(np.float32([[9.0, -9.0]]), np.float32([[1.0, 1.0]]), grid).tolist() == [[3, 0]]
    # all-zero group gets scale 1
    assert O.init_group_scales(np.zeros((1, 128), np.float32), 128, grid)[0, 0] == 1.0


def test_init_logits_bias_on_rtn_level():
    grid = np.array([-1.0, 0.0, 1.0])
    prob = O.Problem(E=1, R=2, C=128, grid=grid, group=128)
    W = np.random.default_rng(2).standard_normal((2, 128)).astype(np.float32) * 0.02
    st = O.init_state(prob, W, np.arange(2), init_bias=2.0)
    codes, margin = O.project(st.logits)
    assert np.array_equal(codes, O.rtn_codes(W, np.repeat(st.scales, 128, 1), grid))
    assert np.all(margin == 2.0)
    assert st.logits.sum() == 2.0 * 256 and np.all(st.m_logits == 0) and np.all(st.m_scales == 0)


def test_kquant2_scales():
    grid = np.linspace(-3.5, 3.5, 8)
    W = (np.random.default_rng(3).standard_normal((3, 512)) * 0.02).astype(np.float32)
    s_eff, d, sc = O.init_kquant2_scales(W, grid)
    sj = np.abs(W).reshape(3, 32, 16).max(2) / np.float32(3.5)
    assert np.all((sc >= 0) & (sc <= 31))
    d_sub = np.repeat(d, 16, axis=1)
    assert np.all(np.abs(s_eff - sj) <= 0.5 * d_sub * (1 + 1e-6))
    np.testing.assert_allclose(d, (sj.reshape(3, 2, 16).max(2) / 31).astype(np.float16).astype(np.float32))
    assert np.array_equal(s_eff, d_sub * sc.astype(np.float32))


def test_project_argmax_ties_lowest():
    l = np.float32([[1.0, 2.0, 3.0], [1.0, 5.0, 3.0], [0.5, 5.0, -1.0]])
    codes, margin = O.project(l)
    assert codes.tolist() == [0, 1, 0]
    assert margin.tolist() == [0.0, 0.0, 0.0]
    codes, margin = O.project(np.float32([[0.0], [2.5], [1.0]]))
    assert codes.tolist() == [1] and margin.tolist() == [1.5]
