"""The C ABI library builds, loads and exports every entry point that
include/rfq.h declares; host-side validation works without a GPU."""
import ctypes
import os
import re

import pytest

from conftest import ROOT


@pytest.fixture(scope="module")
def lib():
    from paper_2608_26581_gb300 import _build, rfq
    _build.build()
    return rfq.load_library()


def _declared():
    src = open(os.path.join(ROOT, "include", "rfq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(rfq_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("rfq_quantize_weight", "rfq_quantize_act", "rfq_linear", "rfq_dequant"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2608_26581_gb300 import rfq
    for n in _declared():
        assert hasattr(lib, n), n
        assert n in rfq.EXPORTED, n


def test_status_strings(lib):
    from paper_2608_26581_gb300 import rfq
    for code, name in rfq.STATUS_NAMES.items():
        assert rfq.rfq_status_string(code).startswith(name)


def test_qtensor_bytes(lib):
    from paper_2608_26581_gb300 import rfq
    assert rfq.rfq_qtensor_bytes(0, 0, 128, 512) == (128 * 256, 128 * 16)
    assert rfq.rfq_qtensor_bytes(0, 1, 130, 512) == (130 * 256, 256 * 16)
    assert rfq.rfq_qtensor_bytes(1, 0, 10, 640) == (10 * 320, 10 * 10 * 4)
    assert rfq.rfq_qtensor_bytes(1, 1, 10, 640) == (10 * 320, 128 * 10 * 4)   # block-major, rows padded
    assert rfq.rfq_qtensor_bytes(2, 0, 10, 640) == (10 * 640 * 2, 0)         # bf16 expansion
    assert rfq.rfq_qtensor_bytes(3, 0, 10, 640) == (10 * 640, 10 * 20)         # MXFP8: a byte per element
    assert rfq.rfq_qtensor_bytes(3, 1, 130, 512) == (130 * 512, 256 * 16)      # MMA scales as MXFP4
    # HiF4: 36 bytes per 64 elements (4.5 bits each)
    cb, sb = rfq.rfq_qtensor_bytes(1, 0, 1, 64)
    assert cb + sb == 36
    with pytest.raises(rfq.RFQError) as e:
        rfq.rfq_qtensor_bytes(0, 1, 128, 96)          # MMA layout needs k % 128
    assert e.value.status == 2
    with pytest.raises(rfq.RFQError) as e:
        rfq.rfq_qtensor_bytes(1, 1, 128, 96)          # HiF4 needs k % 64
    assert e.value.status == 2


def test_workspace_bytes(lib):
    from paper_2608_26581_gb300 import rfq
    assert rfq.rfq_linear_workspace_bytes() >= 4


def test_null_arguments_rejected_before_any_device_work(lib):
    from paper_2608_26581_gb300 import rfq
    assert lib.rfq_quantize_act(None, 1, 32, None, None, None, None, None) == 1
    assert lib.rfq_quantize_weight(None, 32, 16, None, None) == 1
    assert lib.rfq_linear(None, None, None, 0, None, None, 0, None, None) == 1
    assert lib.rfq_dequant(None, None, 0, None) == 1
    qt = rfq._QT(0, 1, 128, 96, 16, 16)           # k not a multiple of 128 for the MMA layout
    assert lib.rfq_quantize_act(ctypes.c_void_p(16), 128, 96, None, ctypes.byref(qt), ctypes.byref(qt),
                                None, None) == 2
    qt = rfq._QT(0, 0, 4, 64, 8, 16)              # misaligned codes pointer
    assert lib.rfq_dequant(ctypes.byref(qt), ctypes.c_void_p(16), 0, None) == 3
    # the checked mode: every call below is rejected on the host, before the device check
    assert lib.rfq_check_finite(None, 4, 64, ctypes.c_void_p(16), None) == 1
    assert lib.rfq_check_finite(ctypes.c_void_p(16), 4, 60, ctypes.c_void_p(16), None) == 2   # k % 8
    assert lib.rfq_check_finite(ctypes.c_void_p(8), 4, 64, ctypes.c_void_p(16), None) == 3    # misaligned
    assert lib.rfq_linear_grouped(None, None, None, 0, None, 1, None, 128, None, 0, None, None) == 1


def test_fused_linear_host_checks(lib):
    """rfq_linear_fused validates its arguments on the host: null pointers,
    K not a multiple of 128, N not a multiple of 16, the phi = AMAX mode it
    does not implement and misaligned pointers are all rejected before any
    device work."""
    from paper_2608_26581_gb300 import rfq
    P = ctypes.c_void_p
    assert lib.rfq_linear_fused(None, 1, 128, None, None, None, 0, None, None) == rfq.RFQ_ERR_INVALID_ARG
    # every call below is rejected on the host: none may reach a launch, since
    # the pointers are not device memory
    wq = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, 256, 128, 16, 16)
    bad_k = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, 256, 96, 16, 16)
    assert lib.rfq_linear_fused(P(16), 4, 96, ctypes.byref(bad_k), None, P(16), 1, P(16), None) == \
        rfq.RFQ_ERR_SHAPE
    bad_n = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, 40, 128, 16, 16)
    assert lib.rfq_linear_fused(P(16), 4, 128, ctypes.byref(bad_n), None, P(16), 1, P(16), None) == \
        rfq.RFQ_ERR_SHAPE
    amax = rfq._FB(rfq.RFQ_FALLBACK_AMAX, 1.0, 128, 256)
    assert lib.rfq_linear_fused(P(16), 4, 128, ctypes.byref(wq), ctypes.byref(amax), P(16), 1, P(16), None) == \
        rfq.RFQ_ERR_UNSUPPORTED
    assert lib.rfq_linear_fused(P(8), 4, 128, ctypes.byref(wq), None, P(16), 1, P(16), None) == \
        rfq.RFQ_ERR_ALIGNMENT


def test_quantize_act_expand_host_checks(lib):
    """rfq_quantize_act_expand validates on the host: the bf16 outputs must be
    present (xr16 exactly when there is a residual), of format RFQ_FMT_BF16,
    shape [M][K] and 16-byte aligned, and the pathway must be HiF4."""
    from paper_2608_26581_gb300 import rfq
    P = ctypes.c_void_p
    M, K = 4, 128
    hq = rfq._QT(rfq.RFQ_FMT_HIF4, rfq.RFQ_SCALE_MMA, M, K, 16, 16)
    mq = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, M, K, 16, 16)
    b16 = rfq._QT(rfq.RFQ_FMT_BF16, 0, M, K, 16, 0)
    b16_shape = rfq._QT(rfq.RFQ_FMT_BF16, 0, M, 64, 16, 0)
    b16_align = rfq._QT(rfq.RFQ_FMT_BF16, 0, M, K, 8, 0)
    none = rfq._FB(rfq.RFQ_FALLBACK_NONE, 0.0, 128, 256)
    r = ctypes.byref
    call = lib.rfq_quantize_act_expand
    assert call(P(16), M, K, None, r(hq), r(hq), None, None, r(b16), None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, None, r(hq), r(hq), None, r(b16), None, None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, r(none), r(hq), None, None, r(b16), r(b16), None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, None, r(mq), r(mq), None, r(b16), r(b16), None) == rfq.RFQ_ERR_UNSUPPORTED
    assert call(P(16), M, K, None, r(hq), r(hq), None, r(b16_shape), r(b16), None) == rfq.RFQ_ERR_SHAPE
    assert call(P(16), M, K, None, r(hq), r(hq), None, r(b16), r(hq), None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, None, r(hq), r(hq), None, r(b16_align), r(b16), None) == rfq.RFQ_ERR_ALIGNMENT


def test_quantize_act_expand_fp8_residual_host_checks(lib):
    """The FP4-to-FP8 form of rfq_quantize_act_expand: X~'s operand is MXFP8
    in the layout of xq, there is no second operand, and the mode must keep
    the residual."""
    from paper_2608_26581_gb300 import rfq
    P = ctypes.c_void_p
    M, K = 4, 128
    x4 = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, M, K, 16, 16)
    x8 = rfq._QT(rfq.RFQ_FMT_MXFP8, rfq.RFQ_SCALE_MMA, M, K, 16, 16)
    x8_row = rfq._QT(rfq.RFQ_FMT_MXFP8, rfq.RFQ_SCALE_ROWMAJOR, M, K, 16, 16)
    b16 = rfq._QT(rfq.RFQ_FMT_BF16, 0, M, K, 16, 0)
    none = rfq._FB(rfq.RFQ_FALLBACK_NONE, 0.0, 128, 256)
    r = ctypes.byref
    call = lib.rfq_quantize_act_expand
    assert call(P(16), M, K, None, r(x4), r(x8), None, r(x8), r(x8), None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, r(none), r(x4), r(x8), None, r(x8), None, None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, None, r(x4), r(x8), None, r(b16), None, None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(P(16), M, K, None, r(x4), r(x8), None, r(x8_row), None, None) == rfq.RFQ_ERR_INVALID_ARG
    # an MXFP4 residual has no operand form to write
    assert call(P(16), M, K, None, r(x4), r(x4), None, r(x8), r(x8), None) == rfq.RFQ_ERR_UNSUPPORTED


def test_fp4_mma_peak_host_checks(lib):
    """rfq_fp4_mma_peak rejects a null workspace or result pointer, a form
    other than 0 / 1, an iteration count outside [1, 2^24] and a misaligned
    workspace on the host (none of these calls reaches a launch)."""
    from paper_2608_26581_gb300 import rfq
    P = ctypes.c_void_p
    flop = ctypes.c_double(0.0)
    r = ctypes.byref
    call = lib.rfq_fp4_mma_peak
    assert call(0, 16, None, r(flop), None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(0, 16, P(16), None, None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(2, 16, P(16), r(flop), None) == rfq.RFQ_ERR_INVALID_ARG
    assert call(1, 0, P(16), r(flop), None) == rfq.RFQ_ERR_SHAPE
    assert call(1, (1 << 24) + 1, P(16), r(flop), None) == rfq.RFQ_ERR_SHAPE
    assert call(0, 16, P(8), r(flop), None) == rfq.RFQ_ERR_ALIGNMENT


def test_noalloc_rejects_before_touching_its_array(lib):
    """rfq_linear_noalloc runs rfq_linear's host checks before it clears its
    shared array: bad arguments return rfq_linear's status (no device work)."""
    from paper_2608_26581_gb300 import rfq
    P = ctypes.c_void_p
    r = ctypes.byref
    assert lib.rfq_linear_noalloc(None, None, None, 0, None, None, 0, None) == rfq.RFQ_ERR_INVALID_ARG
    xq = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, 128, 256, 16, 16)
    wq_bad = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, 40, 256, 16, 16)   # N % 16 != 0
    assert lib.rfq_linear_noalloc(r(xq), None, None, 0, r(wq_bad), P(16), 0, None) == rfq.RFQ_ERR_SHAPE
    assert lib.rfq_linear_noalloc(r(xq), None, None, 0, r(xq), P(8), 0, None) == rfq.RFQ_ERR_ALIGNMENT


def test_debug_bounds_is_the_debug_builds(lib):
    """The normal build carries no bounds checks: rfq_debug_bounds says so."""
    from paper_2608_26581_gb300 import rfq
    st, line = rfq.rfq_debug_bounds()
    assert st == rfq.RFQ_ERR_UNSUPPORTED and line == 0


def test_fp8_activations_with_fp4_weight_host_checks(lib):
    """MXFP8 activations may meet an MXFP4 W~ (multiplied as E2M1 from its
    packed codes): rfq_linear and rfq_linear_grouped reject on the host a W~
    whose codes are not 32-byte aligned (the padded 4-bit copy's rule) and,
    for rfq_linear, K not a multiple of 128; rfq_linear_mixed (which makes
    its padded copy in shared memory) wants the usual 16 bytes; nothing here
    reaches the device check, since the pointers are not device memory."""
    from paper_2608_26581_gb300 import rfq
    P, r = ctypes.c_void_p, ctypes.byref
    M, N, K = 256, 256, 256
    x8 = rfq._QT(rfq.RFQ_FMT_MXFP8, rfq.RFQ_SCALE_MMA, M, K, 32, 32)
    x4 = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, M, K, 32, 32)
    w4_off = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, N, K, 48, 32)     # 16 mod 32
    assert lib.rfq_linear(r(x8), None, None, 256, r(w4_off), P(16), 1, P(16), None) == rfq.RFQ_ERR_ALIGNMENT
    x8k = rfq._QT(rfq.RFQ_FMT_MXFP8, rfq.RFQ_SCALE_MMA, M, 96, 32, 32)
    w4k = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, N, 96, 32, 32)
    assert lib.rfq_linear(r(x8k), None, None, 256, r(w4k), P(16), 1, P(16), None) == rfq.RFQ_ERR_SHAPE
    wg_off = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, 2 * N, K, 48, 32)
    assert lib.rfq_linear_grouped(r(x8), None, None, 256, P(16), 2, r(wg_off), N, P(16), 1, P(16), None) == \
        rfq.RFQ_ERR_ALIGNMENT
    w4_8 = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, N, K, 40, 32)       # 8 mod 16
    assert lib.rfq_linear_mixed(r(x4), r(x8), None, 256, r(w4_8), P(16), 1, P(16), None) == \
        rfq.RFQ_ERR_ALIGNMENT
    # an MXFP8 W~ under MXFP4 activations stays an invalid pairing
    w8 = rfq._QT(rfq.RFQ_FMT_MXFP8, rfq.RFQ_SCALE_MMA, N, K, 32, 32)
    assert lib.rfq_linear(r(x4), None, None, 256, r(w8), P(16), 1, P(16), None) == rfq.RFQ_ERR_INVALID_ARG


def test_linear_host_host_checks(lib):
    """rfq_linear_host validates on the host before any copy is enqueued:
    null buffers, a chunk size that is not a multiple of 128, a residual
    qtensor that does not match the fallback mode, formats other than MXFP4
    and a misaligned x_dev; none of these calls reaches the device."""
    from paper_2608_26581_gb300 import rfq
    P, r = ctypes.c_void_p, ctypes.byref
    M, K, N = 256, 256, 256
    xq = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, M, K, 32, 32)
    wq = rfq._QT(rfq.RFQ_FMT_MXFP4, rfq.RFQ_SCALE_MMA, N, K, 32, 32)
    hq = rfq._QT(rfq.RFQ_FMT_HIF4, rfq.RFQ_SCALE_MMA, M, K, 32, 32)
    none = rfq._FB(rfq.RFQ_FALLBACK_NONE, 0.0, 128, 256)
    call = lib.rfq_linear_host
    H = P(4096)   # stands for a host buffer
    assert call(None, M, K, None, r(wq), H, 0, 0, P(16), r(xq), r(xq), None, P(16), P(16), None) == \
        rfq.RFQ_ERR_INVALID_ARG
    assert call(H, M, K, None, r(wq), None, 0, 0, P(16), r(xq), r(xq), None, P(16), P(16), None) == \
        rfq.RFQ_ERR_INVALID_ARG
    assert call(H, M, K, None, r(wq), H, 0, 100, P(16), r(xq), r(xq), None, P(16), P(16), None) == \
        rfq.RFQ_ERR_SHAPE
    assert call(H, M, K, r(none), r(wq), H, 0, 0, P(16), r(xq), r(xq), None, P(16), P(16), None) == \
        rfq.RFQ_ERR_INVALID_ARG
    assert call(H, M, K, None, r(wq), H, 0, 0, P(16), r(xq), None, None, P(16), P(16), None) == \
        rfq.RFQ_ERR_INVALID_ARG
    assert call(H, M, K, None, r(wq), H, 0, 0, P(16), r(hq), r(hq), None, P(16), P(16), None) == \
        rfq.RFQ_ERR_UNSUPPORTED
    assert call(H, M, K, None, r(wq), H, 0, 0, P(8), r(xq), r(xq), None, P(16), P(16), None) == \
        rfq.RFQ_ERR_ALIGNMENT
