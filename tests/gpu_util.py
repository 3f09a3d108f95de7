"""Helpers shared by the GPU parity tests: device buffers, layout permutations
of the library's scale arrays, and the tolerance checks."""
import numpy as np
import torch

from paper_2608_26581_gb300 import rfq

DEV = "cuda"


def to_dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(DEV).view(torch.bfloat16)


def mma_scale_to_rowmajor(sf_bytes: np.ndarray, rows: int, k: int) -> np.ndarray:
    """Undo the tensor-core scale layout: byte (m, b) sits at
    ((m/128)*(k/128) + b/4)*512 + (m%32)*16 + ((m/32)%4)*4 + b%4."""
    kb = k // 32
    m = np.arange(rows)[:, None]
    b = np.arange(kb)[None, :]
    off = ((m // 128) * (k // 128) + b // 4) * 512 + (m % 32) * 16 + ((m // 32) % 4) * 4 + (b % 4)
    return np.asarray(sf_bytes)[off]


def qtensor_host(q: rfq.QTensor):
    """(codes [rows, k/2] uint8 ([rows, k] for MXFP8), scales in the oracle's
    row-major form)."""
    rows, k = q.rows, q.k
    kc = k if q.fmt == rfq.RFQ_FMT_MXFP8 else k // 2
    codes = q.codes[: rows * kc].cpu().numpy().reshape(rows, kc)
    sf = q.scales.cpu().numpy()
    if q.fmt == rfq.RFQ_FMT_HIF4 and q.scale_layout == rfq.RFQ_SCALE_MMA:
        # block-major [k/64][rows rounded up to 128]
        rp = -(-rows // 128) * 128
        scales = sf[: rp * (k // 64) * 4].view(np.uint32).reshape(k // 64, rp)[:, :rows].T.copy()
    elif q.fmt == rfq.RFQ_FMT_HIF4:
        scales = sf[: rows * (k // 64) * 4].view(np.uint32).reshape(rows, k // 64)
    elif q.scale_layout == rfq.RFQ_SCALE_MMA:
        scales = mma_scale_to_rowmajor(sf, rows, k)
    else:
        scales = sf[: rows * (k // 32)].reshape(rows, k // 32)
    return codes, scales


def check_y(y_gpu: np.ndarray, y_ref: np.ndarray, bf16: bool = False):
    """Y tolerance.  fp32 output: relative Frobenius error <= 1e-5 and max abs
    error <= 1e-3 max|Y|.  bf16 output adds the final rounding to bf16
    (relative 2^-9 per element): relative Frobenius <= 2^-8 and max abs
    <= 1e-3 max|Y| + 2^-8 |Y_ref|."""
    y_gpu = np.asarray(y_gpu, np.float64)
    ref = np.asarray(y_ref, np.float64)
    nrm = np.linalg.norm(ref)
    rel = np.linalg.norm(y_gpu - ref) / max(nrm, 1e-300)
    amax = np.abs(ref).max()
    err = np.abs(y_gpu - ref)
    if bf16:
        ok_abs = np.all(err <= 1e-3 * amax + 2.0 ** -8 * np.abs(ref))
        assert rel <= 2.0 ** -8, f"bf16 rel Frobenius {rel:.3e}"
    else:
        ok_abs = np.all(err <= 1e-3 * amax)
        assert rel <= 1e-5, f"rel Frobenius {rel:.3e}"
    assert ok_abs, f"max abs err {err.max():.3e} vs max|Y| {amax:.3e}"
    return rel


# Canary guard bytes: buffers the kernels write are allocated with GUARD
# extra bytes filled with CANARY after their end, and every guard is checked
# after the test (a write past the end of an output shows up there).
CANARY = 0xA5
GUARD = 256
_guarded = []


def guarded_bytes(nbytes: int) -> torch.Tensor:
    """A uint8 device buffer of nbytes followed by GUARD canary bytes; the
    returned tensor is the nbytes payload (16-byte aligned)."""
    base = torch.empty(nbytes + GUARD, dtype=torch.uint8, device=DEV)
    base[nbytes:].fill_(CANARY)
    _guarded.append((base, nbytes))
    return base[:nbytes]


def guarded_empty(shape, dtype) -> torch.Tensor:
    n = int(np.prod(shape)) * torch.empty(0, dtype=dtype).element_size()
    return guarded_bytes(n).view(dtype).view(*shape)


def guarded_full(shape, value, dtype) -> torch.Tensor:
    t = guarded_empty(shape, dtype)
    t.fill_(value)
    return t


def guarded_qtensor(fmt: int, scale_layout: int, rows: int, k: int, device=DEV) -> rfq.QTensor:
    cb, sb = rfq.rfq_qtensor_bytes(fmt, scale_layout, rows, k)
    return rfq.QTensor(fmt, scale_layout, rows, k, guarded_bytes(max(cb, 16)), guarded_bytes(max(sb, 16)))


def check_guards():
    """Every guard allocated since the last check still holds CANARY."""
    torch.cuda.synchronize()
    bad = [(n, int((b[n:] != CANARY).sum())) for b, n in _guarded if not bool((b[n:] == CANARY).all())]
    _guarded.clear()
    assert not bad, f"bytes past the end of an output buffer were written: {bad}"
