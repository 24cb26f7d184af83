"""Small test utilities: bf16 bit conversion and a dense scipy formulation.

The dense formulation builds the whole masked logit matrix with a matrix
product and hands it to scipy's logsumexp/softmax; it is an independent
construction used only to pin the row-by-row oracle on tiny inputs.
"""
import numpy as np


def f32_to_bf16_bits(x) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest-even) and return the bit patterns."""
    a = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = a.view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return r.astype(np.uint16).reshape(a.shape)


def bf16_bits_to_f64(b) -> np.ndarray:
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def random_bf16(rng, shape, scale=1.0):
    return f32_to_bf16_bits(rng.standard_normal(shape) * scale)


def dense_reference(q, k, v, cu_q, cu_k, Hq, Hkv, scale):
    """Masked dense attention through scipy.special; q, k, v are bf16 bit arrays."""
    from scipy.special import logsumexp, softmax
    qf, kf, vf = bf16_bits_to_f64(q), bf16_bits_to_f64(k), bf16_bits_to_f64(v)
    G = Hq // Hkv
    kx = np.repeat(kf, G, axis=1)  # [total_k, Hq, d]: kv head g serves query heads gG..gG+G-1
    vx = np.repeat(vf, G, axis=1)
    total_q, _, d = qf.shape
    o = np.zeros((total_q, Hq, d))
    lse = np.full((total_q, Hq), -np.inf)
    for s in range(len(cu_q) - 1):
        q0, q1, k0, k1 = cu_q[s], cu_q[s + 1], cu_k[s], cu_k[s + 1]
        Lq, Lk = q1 - q0, k1 - k0
        if Lq == 0:
            continue
        visible = np.tril(np.ones((Lq, Lk), dtype=bool), k=Lk - Lq)
        for h in range(Hq):
            logits = scale * (qf[q0:q1, h, :] @ kx[k0:k1, h, :].T)
            logits = np.where(visible, logits, -np.inf)
            rows = visible.any(axis=1)
            if not rows.any():
                continue
            lse[q0:q1, h][rows] = logsumexp(logits[rows], axis=1)
            w = softmax(logits[rows], axis=1)
            o[q0:q1, h, :][rows] = w @ vx[k0:k1, h, :]
    return o, lse
