"""Comparison rules between the CUDA path and the CPU oracle.

Tolerances (stated once here, used by every parity test):

* rotated rows X~ (fp32): per row ||g - o||_2 <= 1e-5 ||o||_2 and every
  element |g - o| <= 1e-5 * max_k |o[k]|.  The oracle's rotation is exact and
  rounded once; the GPU's butterflies round after each of log2(b) stages, so
  each element carries at most about log2(b) * 2^-24 relative error of the
  block's magnitude, well inside 1e-5.
* scales s = absmax / 7: equal, or within 2 ulp where the abs-max element
  itself differs in its last bits (relative 2.5e-7).
* INT4 codes: equal, except entries off by exactly one where the oracle's
  ratio X~ / s lies within 1e-4 of a half-integer (a rounding tie at fp32
  resolution); at most max(1, 1e-4 * n) such entries.
* integer accumulators: bit-exact when the GPU GEMM is fed the oracle's codes.
* outputs Y: ||Y - y64||_F <= 1e-2 ||y64||_F against the oracle's fp64
  dequantized product; when fed identical codes and scales also elementwise
  |Y - y64| <= u * |y64| + 1e-6 * (|acc s_x s_w / b| + |bias|) + tiny, with u
  the output format's half-ulp (2^-11 fp16, 2^-8 bf16).
"""
import numpy as np


def check_rot(g, o):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    rowmax = np.max(np.abs(o), axis=1, keepdims=True)
    err = np.abs(g - o)
    assert np.all(err <= 1e-5 * rowmax + 1e-30), float(np.max(err / (rowmax + 1e-30)))
    num = np.linalg.norm(g - o, axis=1)
    den = np.linalg.norm(o, axis=1)
    assert np.all(num <= 1e-5 * den + 1e-30)


def check_scales(g, o):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    assert np.all(np.abs(g - o) <= 2.5e-7 * np.abs(o)), float(np.max(np.abs(g - o)))


def check_codes(gc, oc, o_rot, o_s):
    gc = np.asarray(gc, np.int64)
    oc = np.asarray(oc, np.int64)
    bad = gc != oc
    n_bad = int(np.count_nonzero(bad))
    if n_bad == 0:
        return 0
    assert np.all(np.abs(gc[bad] - oc[bad]) == 1), "codes differ by more than one"
    s = np.asarray(o_s, np.float64)[:, None] * np.ones_like(np.asarray(o_rot, np.float64))
    ratio = np.asarray(o_rot, np.float64)[bad] / s[bad]
    dist = np.abs(np.abs(ratio - np.floor(ratio)) - 0.5)
    assert np.all(dist <= 1e-4), "off-by-one code away from a rounding tie"
    assert n_bad <= max(1, int(1e-4 * gc.size)), n_bad
    return n_bad


def check_output_frobenius(y, y64, tol=1e-2):
    y = np.asarray(y, np.float64)
    y64 = np.asarray(y64, np.float64)
    rel = np.linalg.norm(y - y64) / max(np.linalg.norm(y64), 1e-300)
    assert rel <= tol, rel
    return rel


def check_output_elementwise(y, y64, acc, s_x, s_w, b, bias, dtype):
    y = np.asarray(y, np.float64)
    y64 = np.asarray(y64, np.float64)
    prod = np.abs(np.asarray(acc, np.float64) * np.asarray(s_x, np.float64)[:, None]
                  * np.asarray(s_w, np.float64)[None, :] / b)
    bb = 0.0 if bias is None else np.abs(np.asarray(bias, np.float64))[None, :]
    u = 2.0 ** -11 if dtype == "f16" else 2.0 ** -8
    tiny = 2.0 ** -24 if dtype == "f16" else 2.0 ** -126
    tol = u * np.abs(y64) + 1e-6 * (prod + bb) + tiny
    err = np.abs(y - y64)
    assert np.all(err <= tol), float(np.max(err - tol))
