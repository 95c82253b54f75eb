"""CPU oracle for the Hadamard-domain INT8 convolution (HaTQ). TEST
INFRASTRUCTURE ONLY: tests, the smoke check and the benchmark's CPU-baseline
leg may import it; the CUDA path never does, and nothing here is shared with
it (the two are written independently and meet only on the seeded inputs).

Plain, slow and literal: dense Sylvester matrices, matrix-form transforms,
scalar quantizers, a nested-loop direct convolution (conv_ref.c), fp64 for
real arithmetic and int64 (or Python integers) for integer arithmetic.

Section/equation names refer to the HaTQ paper ("Hadamard-Domain Model
Quantization for Learned Image Coding") and its supplementary material.

Readings the paper leaves open (the same list is kept with the design notes):
  R1 transform order: a block-diagonal Sylvester transform I_{C/hb} (x) H_hb
     along the channel axis (orthogonal, so the DH/WH identities hold), not the
     single Paley/Kronecker order m(C) of Eq. (hadamard_order).
  R2 round(.) is round-half-to-even everywhere (rint for reals; for a shift
     by 2^n the exact rational v / 2^n rounded half to even).
  R3 the multiplier/shift pair (M, n) of Eq. (integer_fixed_point_scale):
     the largest shared n in [0, 62] such that every M_c = rint(rho_c 2^n) is
     below 2^31 and max_c(M_c A_c) * g_out * g_next < 2^62, with A_c the
     worst-case |accumulator| of channel c and g the gains (block sizes) of the
     unnormalized transforms; fewer than 16 bits in max_c M_c is an error. The
     INT8-entry activation requantizer (a 32-bit computation) takes the bound
     M 127 hb < 2^30 instead of 2^62 and a 15-bit precision floor.
  R4 symmetric INT8 range [-127, 127]; a zero range gives scale 1.
  R5 bias enters the int32 accumulator before M (.) and before H_out.
  R6 fixed summation order for real-valued transforms: for output j,
     acc = 0; acc += H[i][j] * x_i for i = 0..hb-1; then acc / sqrt(hb).

  R7 non-homogeneous activations (SiLU, GELU; GDN, IGDN on the channel
     vector) take the two-step transition of the supplementary's general
     nonlinearities: both multiplier/shift pairs by R3, phi_int in fp64
     (math-library exp / erf, a table for the elementwise ones) rounded by R2.
  R8 the range-expansion statistic is decided on the INT8 codes a layer
     receives, exactly: max|H~ x|^2 > hb max|x|^2.
  R9 Paley constructions are taken over primes q only. Where an order has
     several constructions (the paper fixes none) the matrix is the first of:
     Sylvester (a power of two), Paley-I (q = m - 1), Paley-II (q = m / 2 - 1),
     else H~_a (x) H~_(m/a) with a the smallest supported order >= 2 whose
     cofactor m / a is supported, each factor by the same rule.
  R10 transposed convolutions use the same prepared weights (DH / WH along
     C_in / C_out) as a scatter; the integer transition is unchanged.
  R11 dynamic affine activations: unsigned 8-bit codes (q_min 0, q_max 255),
     a zero range gives (s, z) = (1, 0), the input-side operand (T x for DH)
     is quantized and padding is a centred zero.
  R21 phi_int for GDN / IGDN (Eq. supp_general_activation) in integers:
     G_ij = rint(gamma_ij s_z^2 2^e), B_i = max(1, rint(beta_i 2^e)) with the
     largest e such that max G <= 511 and max_i (B_i + 127^2 sum_j G_ij) < 2^31;
     D_i = B_i + sum_j G_ij z_j^2 (exact). GDN: X_i = R |z_i| / sqrt(D_i) with
     R^2 = (s_z / s_u)^2 2^e; IGDN: X_i = R |z_i| sqrt(D_i) with
     R^2 = (s_z / s_u)^2 2^-e. R^2 ~ P / 2^t (largest t keeping the tests below
     in 63 bits, P >= 2^15). |u_i| = min(127, round(X_i)) with ties away from
     zero, decided exactly: the largest k with (2k - 1)^2 D_i 2^t <= 4 P z_i^2
     (GDN) or (2k - 1)^2 2^t <= 4 P z_i^2 D_i (IGDN); u_i takes the sign of z_i.

Pins (tests/test_oracle_pins.py) hold every function to something other
than itself: closed forms, the paper's printed values, brute force and exact
rational arithmetic. R2 and R3 are readings (the paper fixes no rounding
convention and no rule for n); what they define is pinned against exact
rationals: the shift equals the exact rational v / 2^n rounded half to even,
and (M, n) is the largest admissible n with |M - rho 2^n| <= 1/2.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from fractions import Fraction

import numpy as np

QMAX = 127                      # q_max^s = 2^(b-1) - 1 for b = 8, Eq. (symmetric_q)

# --------------------------------------------------------------------------
# Hadamard matrices: Eq. (supp_sylvester), Eq. (hadamard_properties)
# --------------------------------------------------------------------------


def sylvester(m: int) -> np.ndarray:
    """Unnormalized Sylvester Hadamard matrix H~_m by the recursion
    H~_1 = [1], H~_2m = [[H~_m, H~_m], [H~_m, -H~_m]] (Eq. supp_sylvester)."""
    if m < 1 or (m & (m - 1)) != 0:
        raise ValueError("Sylvester order must be a power of two")
    H = np.ones((1, 1), dtype=np.int64)
    while H.shape[0] < m:
        H = np.block([[H, H], [H, -H]])
    return H


# --------------------------------------------------------------------------
# Paper-exact orders (Supp. Hadamard construction): Paley-I / Paley-II and
# Kronecker products, Eq. (hadamard_order), padded transforms of Eq.
# (supp_padded_transforms). Reading: q is restricted to primes (the paper
# allows prime powers, whose finite-field arithmetic is not built here).
# --------------------------------------------------------------------------


def _is_prime(q: int) -> bool:
    if q < 2:
        return False
    f = 2
    while f * f <= q:
        if q % f == 0:
            return False
        f += 1
    return True


def _jacobsthal(q: int) -> np.ndarray:
    """Q[i, j] = chi(j - i) with chi the quadratic character modulo the prime q."""
    squares = {(x * x) % q for x in range(1, q)}
    chi = np.array([0] + [1 if a in squares else -1 for a in range(1, q)], dtype=np.int64)
    idx = (np.arange(q)[None, :] - np.arange(q)[:, None]) % q
    return chi[idx]


def paley1(q: int) -> np.ndarray:
    """Paley-I Hadamard matrix of order q + 1, q a prime with q = 3 (mod 4):
    H = I + S with S = [[0, 1^T], [-1, Q]] (S antisymmetric)."""
    if not _is_prime(q) or q % 4 != 3:
        raise ValueError("Paley-I needs a prime q = 3 (mod 4)")
    Q = _jacobsthal(q)
    S = np.zeros((q + 1, q + 1), dtype=np.int64)
    S[0, 1:] = 1
    S[1:, 0] = -1
    S[1:, 1:] = Q
    return np.eye(q + 1, dtype=np.int64) + S


def paley2(q: int) -> np.ndarray:
    """Paley-II Hadamard matrix of order 2 (q + 1), q a prime with q = 1 (mod 4):
    the symmetric conference matrix C = [[0, 1^T], [1, Q]] gives
    H = C (x) [[1, 1], [1, -1]] + I (x) [[1, -1], [-1, -1]]."""
    if not _is_prime(q) or q % 4 != 1:
        raise ValueError("Paley-II needs a prime q = 1 (mod 4)")
    Q = _jacobsthal(q)
    Cm = np.zeros((q + 1, q + 1), dtype=np.int64)
    Cm[0, 1:] = 1
    Cm[1:, 0] = 1
    Cm[1:, 1:] = Q
    A = np.array([[1, 1], [1, -1]], dtype=np.int64)
    B = np.array([[1, -1], [-1, -1]], dtype=np.int64)
    return np.kron(Cm, A) + np.kron(np.eye(q + 1, dtype=np.int64), B)


def _base_orders(limit: int) -> dict:
    """Orders <= limit with a direct construction, each with its constructor by
    reading R9: Sylvester for a power of two, else Paley-I (q = m - 1 a prime,
    q = 3 mod 4), else Paley-II (q = m / 2 - 1 a prime, q = 1 mod 4)."""
    out = {}
    for m in range(1, limit + 1):
        if m & (m - 1) == 0:
            out[m] = ("sylvester", m)
        elif _is_prime(m - 1) and (m - 1) % 4 == 3:
            out[m] = ("paley1", m - 1)
        elif m % 2 == 0 and _is_prime(m // 2 - 1) and (m // 2 - 1) % 4 == 1:
            out[m] = ("paley2", m // 2 - 1)
    return out


_ORDERS_CACHE = {}


def supported_orders(limit: int = 1024) -> dict:
    """The set M_H of supported orders <= limit: base orders and Kronecker
    products of supported orders, each with its recipe under reading R9 (a
    nested tuple; recipes only, no matrices), cached per limit."""
    if limit in _ORDERS_CACHE:
        return dict(_ORDERS_CACHE[limit])
    base = _base_orders(limit)
    members = set(base)
    changed = True
    while changed:
        changed = False
        for a in sorted(members):
            for b in sorted(members):
                if a >= 2 and b >= 2 and a * b <= limit and a * b not in members:
                    members.add(a * b)
                    changed = True
    orders = {}
    for m in sorted(members):
        if m in base:
            orders[m] = base[m]
        else:
            a = min(f for f in members if f >= 2 and m % f == 0 and m // f in members)
            orders[m] = ("kron", a, m // a)
    _ORDERS_CACHE[limit] = dict(orders)
    return orders


def hadamard_of_order(m: int, orders: dict = None) -> np.ndarray:
    """The unnormalized Hadamard matrix of a supported order m (reading R9)."""
    orders = orders or supported_orders(max(1024, m))
    if m not in orders:
        raise ValueError(f"order {m} is not supported")
    r = orders[m]
    if r[0] == "sylvester":
        return sylvester(m)
    if r[0] == "paley1":
        return paley1(r[1])
    if r[0] == "paley2":
        return paley2(r[1])
    return np.kron(hadamard_of_order(r[1], orders), hadamard_of_order(r[2], orders))


def hadamard_order(c: int, limit: int = 4096) -> int:
    """m(C) of Eq. (hadamard_order): the smallest supported order >= 4 ceil(C / 4)."""
    c4 = 4 * ((c + 3) // 4)
    orders = supported_orders(limit)
    return min(m for m in orders if m >= c4)


def padded_transforms(c: int):
    """T_in = P_C H_m and T_out = P_C H_m^T of Eq. (supp_padded_transforms),
    with H_m = H~_m / sqrt(m) and P_C = [I_C 0]: [C, m] fp64 each."""
    m = hadamard_order(c)
    H = hadamard_of_order(m).astype(np.float64) / math.sqrt(m)
    return H[:c, :], H.T[:c, :]


def blockdiag_transform(c: int, hb: int) -> np.ndarray:
    """Normalized block-diagonal transform T = I_{c/hb} (x) H_hb (reading R1),
    H_hb = H~_hb / sqrt(hb) (Eq. hadamard_properties). Dense fp64 [c, c]."""
    if c % hb:
        raise ValueError("channel count must be a multiple of the block")
    H = sylvester(hb).astype(np.float64) / math.sqrt(hb)
    return np.kron(np.eye(c // hb), H)


def _blocks(x: np.ndarray, hb: int) -> np.ndarray:
    c = x.shape[-1]
    if c % hb:
        raise ValueError("channel count must be a multiple of the block")
    return x.reshape(x.shape[:-1] + (c // hb, hb))


def transform_int(x: np.ndarray, hb: int) -> np.ndarray:
    """Unnormalized integer transform along the last axis, block by block:
    y_blk = H~_hb x_blk, exact in int64 (the integer transforms of the
    integer basis conversions, Table integer_transitions)."""
    x = np.asarray(x, dtype=np.int64)
    if hb <= 1:
        return x.copy()
    H = sylvester(hb)
    y = _blocks(x, hb) @ H.T            # y_j = sum_i H~[j, i] x_i
    return y.reshape(x.shape)


def transform_real(x: np.ndarray, hb: int, normalize: bool = True) -> np.ndarray:
    """Real-valued transform along the last axis in the fixed order of
    reading R6: y_j = (sum_{i=0}^{hb-1} H~[i][j] x_i) / sqrt(hb)."""
    x = np.asarray(x, dtype=np.float64)
    if hb <= 1:
        return x.copy()
    H = sylvester(hb).astype(np.float64)
    xb = _blocks(x, hb)
    acc = np.zeros_like(xb)
    for i in range(hb):
        acc += H[i][None, :] * xb[..., i:i + 1]
    if normalize:
        acc = acc / math.sqrt(hb)
    return acc.reshape(x.shape)


def transform_order_real(x: np.ndarray, m: int) -> np.ndarray:
    """x T_in with T_in = P_C H_m of Eq. (supp_padded_transforms): the last
    axis (C channels) is zero-padded to the order m >= C and multiplied by the
    normalized H_m of reading R9, in the fixed order of reading R6:
    y_j = (sum_{i=0}^{C-1} H~[i][j] x_i) / sqrt(m). Returns [..., m] fp64."""
    x = np.asarray(x, dtype=np.float64)
    c = x.shape[-1]
    if m < c:
        raise ValueError("the order must be at least the channel count")
    H = hadamard_of_order(m).astype(np.float64)
    acc = np.zeros(x.shape[:-1] + (m,))
    for i in range(c):
        acc += H[i][None, :] * x[..., i:i + 1]
    return acc / math.sqrt(m)


def transform_order_int(x_i8, m: int) -> np.ndarray:
    """Unnormalized integer transform of the zero-padded channel vector,
    y_j = sum_{i<C} H~[i][j] x_i, exact in int64: [..., m]."""
    x = np.asarray(x_i8, dtype=np.int64)
    H = hadamard_of_order(m)
    return x @ H[:x.shape[-1], :]


# --------------------------------------------------------------------------
# Quantizers: Eq. (symmetric_q), reading R2/R4
# --------------------------------------------------------------------------


def symmetric_scale(x) -> float:
    """s = ||x||_inf / q_max (Eq. symmetric_q); 1.0 for an all-zero tensor (R4)."""
    m = float(np.max(np.abs(np.asarray(x, dtype=np.float64)))) if np.size(x) else 0.0
    return m / QMAX if m > 0 else 1.0


def quantize_sym(x, s: float) -> np.ndarray:
    """x_int = clamp(round(x / s), -q_max, q_max) (Eq. symmetric_q)."""
    q = np.rint(np.asarray(x, dtype=np.float64) / s)
    return np.clip(q, -QMAX, QMAX).astype(np.int64)


def rshift_rne(v, n: int) -> np.ndarray:
    """round(v / 2^n) for integer v, ties to even (R2), exact in int64."""
    v = np.asarray(v, dtype=np.int64)
    if n == 0:
        return v.copy()
    q = v >> n                                    # floor(v / 2^n)
    r = v - (q << n)                              # in [0, 2^n)
    half = np.int64(1) << (n - 1)
    up = (r > half) | ((r == half) & ((q & 1) == 1))
    return q + up.astype(np.int64)


def fixed_point(rho, a_bound, gain: int = 1, prod_bits: int = 62, min_bits: int = 16):
    """Multiplier/shift pair of Eqs. (fixed_point_scale, integer_fixed_point_scale)
    under reading R3. rho: per-channel real ratios (> 0); a_bound: per-channel
    bound on |input| of the multiplication; gain: product of the unnormalized
    transform gains applied after M (.); prod_bits: the products M a gain stay
    below 2^prod_bits (62 for the 64-bit epilogue, 30 for the 32-bit activation
    requantizer); min_bits: the least multiplier precision (16, and 15 for
    the activation requantizer, whose 32-bit bound leaves 15 bits at hb = 256).
    Returns (M int64 array, n)."""
    rho = np.asarray(rho, dtype=np.float64)
    a_bound = [int(a) for a in np.asarray(a_bound).ravel()]
    if np.any(rho < 0) or not np.all(np.isfinite(rho)):
        raise ValueError("scale ratios must be finite and nonnegative")
    for n in range(62, -1, -1):
        M = [int(np.rint(math.ldexp(float(r), n))) for r in rho]
        if max(M) >= 2 ** 31:
            continue
        worst = max(m * a for m, a in zip(M, a_bound)) * int(gain)
        if worst >= 2 ** prod_bits:
            continue
        if max(M) < 2 ** (min_bits - 1):
            raise OverflowError(f"fewer than {min_bits} bits of multiplier precision")
        return np.array(M, dtype=np.int64), n
    raise OverflowError("no shift satisfies the multiplier and overflow bounds")


def round_half_even_fraction(f: Fraction) -> int:
    fl = f.numerator // f.denominator
    r = f - fl
    if r > Fraction(1, 2) or (r == Fraction(1, 2) and fl % 2 == 1):
        return fl + 1
    return fl


def dynamic_multiplier(maxy: int, hb: int):
    """(M, n) for the dynamic INT8-entry quantizer: rho = 127 / max|y| as an
    exact rational, M = round(rho 2^n) half to even, n by reading R3 with the
    activation requantizer's 32-bit product bound M 127 hb < 2^30."""
    if maxy <= 0:
        return 0, 0
    for n in range(62, -1, -1):
        M = round_half_even_fraction(Fraction(QMAX << n, maxy))
        if M >= 2 ** 31 or M * QMAX * hb >= 2 ** 30:
            continue
        if M < 2 ** 14:
            raise OverflowError("fewer than 15 bits of multiplier precision")
        return M, n
    raise OverflowError("no shift satisfies the bounds")


# --------------------------------------------------------------------------
# Weight preparation (offline): DH Eq. (double_hadamard_quantization),
# WH Eq. (supp_padded_wh_parameters), bias Eq. (supp_bias_quantization),
# requant Eq. (integer_fixed_point_scale) with Table integer_transitions.
# --------------------------------------------------------------------------


def transform_weights(w_ohwi, b, form: str, hb_in: int, hb_out: int):
    """Hadamard-domain weights and bias (fp64).
    DH: W' = W (I_{KhKw} (x) T_in): every tap's C_in vector is transformed
        (Eq. input_hadamard_transform); bias unchanged.
    WH: W_bar = T_out^T W along C_out, b_bar = b T_out
        (Eq. supp_padded_wh_parameters)."""
    w = np.asarray(w_ohwi, dtype=np.float64)
    bb = np.zeros(w.shape[0]) if b is None else np.asarray(b, dtype=np.float64)
    if form == "DH":
        return transform_real(w, hb_in), bb.copy()
    if form == "WH":
        wt = np.moveaxis(w, 0, -1)                    # [kh, kw, ci, co]
        wbar = np.moveaxis(transform_real(wt, hb_out), -1, 0)
        return wbar, transform_real(bb, hb_out)
    raise ValueError(form)


class Prepared:
    """One prepared layer: INT8 weights, per-channel scales, bias codes and
    fixed-point requant parameters, in the Hadamard domain of its form."""

    def __init__(self, **kw):
        self.__dict__.update(kw)


GENERAL_ACTS = ("silu", "gelu")
VECTOR_ACTS = ("gdn", "igdn")


def phi(kind: str, v: float) -> float:
    """The non-homogeneous activations of Sec. general nonlinearities, fp64
    (math-library exp / erf): SiLU v / (1 + e^-v), GELU v (1 + erf(v / sqrt 2)) / 2."""
    if kind == "silu":
        return v / (1.0 + math.exp(-v))
    if kind == "gelu":
        return 0.5 * v * (1.0 + math.erf(v / math.sqrt(2.0)))
    raise ValueError(kind)


def activation_lut(kind: str, s_z: float, s_u: float) -> np.ndarray:
    """phi_int of Eq. (supp_general_activation) as an integer lookup table over
    the preactivation codes z = -127..127 (index z + 127):
    u = clamp(round(phi(s_z z) / s_u), -127, 127), rounded half to even (R2)."""
    s_z = float(np.float32(s_z))
    s_u = float(np.float32(s_u))
    out = np.zeros(255, dtype=np.int64)
    for i, z in enumerate(range(-QMAX, QMAX + 1)):
        out[i] = min(max(int(round(phi(kind, s_z * z) / s_u)), -QMAX), QMAX)
    return out


def prepare_layer(w_ohwi, b, form: str, hb_in: int, hb_out: int, s_x: float,
                  s_y: float, act: str, hb_next: int, out_f32: bool,
                  stride: int, pad: int, s_z: float = None, s_u: float = None,
                  order_in: int = 0, gdn_beta=None, gdn_gamma=None) -> Prepared:
    """Offline preparation of one layer (Sec. deployment realization).
    s_x: scale of the INT8 operand this layer consumes; s_y: scale of the
    INT8 operand the next layer consumes (or of this layer's output).
    A non-homogeneous act ('silu', 'gelu'; 'gdn', 'igdn' with gdn_beta,
    gdn_gamma) takes the two-step transition of Sec. general nonlinearities
    with preactivation scale s_z and activation scale s_u. order_in > 0 (DH only): the input side takes the paper's
    single order m = order_in instead of blocks, W' = W (I (x) P_C H_m)
    (Eqs. supp_padded_transforms, supp_padded_dh); the layer then consumes an
    operand of m channels."""
    s_x = float(np.float32(s_x))
    s_y = float(np.float32(s_y))
    if order_in:
        if form != "DH":
            raise ValueError("a paper-order input transform belongs to a DH layer")
        wprime = transform_order_real(w_ohwi, order_in)
        bbar = np.zeros(wprime.shape[0]) if b is None else np.asarray(b, dtype=np.float64).copy()
    else:
        wprime, bbar = transform_weights(w_ohwi, b, form, hb_in, hb_out)
    co = wprime.shape[0]
    flat = wprime.reshape(co, -1)
    maxabs = np.max(np.abs(flat), axis=1)
    s_w = np.where(maxabs > 0, maxabs / QMAX, 1.0)               # channel-wise Eq. symmetric_q
    w_int = np.clip(np.rint(flat / s_w[:, None]), -QMAX, QMAX).astype(np.int64)
    s_a = s_x * s_w                                              # Eq. accumulator_scale
    b_int = np.rint(bbar / s_a).astype(np.int64)                 # Eq. supp_bias_quantization
    g_out = math.sqrt(hb_out) if form == "WH" else 1.0           # Table integer_transitions
    g_in = math.sqrt(hb_next) if hb_next else 1.0
    a_bound = QMAX * np.sum(np.abs(w_int), axis=1) + np.abs(b_int)
    if int(np.max(a_bound)) >= 2 ** 31:
        raise OverflowError("int32 accumulator bound exceeded")
    prep = Prepared(form=form, hb_in=hb_in, hb_out=hb_out if form == "WH" else 0, order_in=order_in,
                    hb_next=hb_next, act=act, out_f32=out_f32, stride=stride, pad=pad,
                    s_x=s_x, s_y=s_y, s_w=s_w, b_int=b_int,
                    w_int=w_int.reshape(wprime.shape).astype(np.int8),
                    a_bound=a_bound, wprime=wprime, bbar=bbar)
    if act in GENERAL_ACTS or act in VECTOR_ACTS:
        if out_f32:
            raise ValueError("the general transition emits INT8 codes")
        s_z = float(np.float32(s_z))
        s_u = float(np.float32(s_u))
        # Eq. supp_general_output_scale: s_A,c / (gamma_out s_z) ~ M_out / 2^n_out, M before H_out
        prep.M, prep.n = fixed_point(s_a / (g_out * s_z), a_bound, hb_out if form == "WH" else 1)
        prep.lut = activation_lut(act, s_z, s_u) if act in GENERAL_ACTS else None
        prep.gdn = gdn_params(gdn_beta, gdn_gamma, s_z, s_u, act == "igdn") if act in VECTOR_ACTS else None
        # Eq. supp_general_input_scale: s_u / (gamma_in,next s_x,next) ~ M_in / 2^n_in
        M_in, n_in = fixed_point([s_u / (g_in * s_y)], [QMAX], hb_next if hb_next else 1)
        prep.M_in, prep.n_in = int(M_in[0]), n_in
        prep.s_z, prep.s_u = s_z, s_u
        return prep
    if out_f32:
        prep.deq = s_a / g_out
        prep.M, prep.n = None, 0
    else:
        alpha = g_out * g_in
        rho = s_a / (alpha * s_y)                                # Eq. integer_fixed_point_scale
        gain = (hb_out if form == "WH" else 1) * (hb_next if hb_next else 1)
        prep.M, prep.n = fixed_point(rho, a_bound, gain)
        prep.rho = rho
    return prep


# --------------------------------------------------------------------------
# Activation transform + quantize (online): Eqs. (double_hadamard_quantization,
# symmetric_q); INT8 entry uses the integer input transform and fixed-point
# rescaling of Eq. (supp_general_input_transition) with M^in, n^in.
# --------------------------------------------------------------------------


def quantize_act_f16(x, hb: int, s_x: float) -> np.ndarray:
    """FP16 entry: codes of Q_a(X H_in): clamp(rint((H~ x)_j / (sqrt(hb) s_x)))."""
    y = transform_real(np.asarray(x, dtype=np.float64), hb, normalize=False)
    return np.clip(np.rint(y / (math.sqrt(hb) * float(np.float32(s_x)))), -QMAX, QMAX).astype(np.int8)


def act_multiplier(hb: int, s_in: float, s_x: float):
    """(M_q, n_q) with M_q / 2^n_q ~ s_in / (sqrt(hb) s_x), bound |y| <= 127 hb,
    products M_q |y| below 2^30 (reading R3, 32-bit activation requantizer)."""
    rho = float(np.float32(s_in)) / (math.sqrt(hb) * float(np.float32(s_x)))
    M, n = fixed_point([rho], [QMAX * hb], 1, prod_bits=30, min_bits=15)
    return int(M[0]), n


def quantize_act_i8(x_i8, hb: int, s_in: float, s_x: float) -> np.ndarray:
    """INT8 entry: y = H~ x (exact), codes = clamp(round(M_q y / 2^n_q))."""
    M, n = act_multiplier(hb, s_in, s_x)
    y = transform_int(x_i8, hb)
    return np.clip(rshift_rne(M * y, n), -QMAX, QMAX).astype(np.int8)


def quantize_act_order_i8(x_i8, m: int, s_in: float, s_x: float) -> np.ndarray:
    """INT8 entry into the paper's order-m basis (the activation side of
    Eq. supp_padded_dh): y = x_int P_C H~_m exactly, codes =
    clamp(round(M_q y / 2^n_q)) with M_q / 2^n_q ~ s_in / (sqrt(m) s_x) by
    reading R3 over the bound |y| <= 127 C. Returns [..., m] int8."""
    x = np.asarray(x_i8, dtype=np.int64)
    c = x.shape[-1]
    rho = float(np.float32(s_in)) / (math.sqrt(m) * float(np.float32(s_x)))
    M, n = fixed_point([rho], [QMAX * c], 1)
    y = transform_order_int(x, m)
    return np.clip(rshift_rne(int(M[0]) * y, n), -QMAX, QMAX).astype(np.int8)


def quantize_act_dynamic_i8(x_i8, hb: int, s_in: float):
    """Dynamic per-tensor scale (PTQ, Sec. network-wise PTQ): s from the
    transformed tensor's max-abs, then the INT8 entry quantizer. Returns
    (codes, s_used) with s_used = s_in max|H~x| / (sqrt(hb) 127) (fp64 -> fp32)."""
    y = transform_int(x_i8, hb)
    maxy = int(np.max(np.abs(y))) if y.size else 0
    if maxy == 0:
        return np.zeros(y.shape, dtype=np.int8), 1.0
    M, n = dynamic_multiplier(maxy, hb)
    codes = np.clip(rshift_rne(M * y, n), -QMAX, QMAX).astype(np.int8)
    s_used = float(np.float32(float(np.float32(s_in)) * maxy / (math.sqrt(hb) * QMAX)))
    return codes, s_used


def quantize_act_dynamic_f16(x, hb: int):
    """Dynamic FP16 entry: s = max|H x| / 127; returns (codes, s_used)."""
    y = transform_real(np.asarray(x, dtype=np.float64), hb, normalize=False)
    m = float(np.max(np.abs(y))) if y.size else 0.0
    if m == 0.0:
        return np.zeros(y.shape, dtype=np.int8), 1.0
    codes = np.clip(np.rint(y * (QMAX / m)), -QMAX, QMAX).astype(np.int8)
    return codes, m / (math.sqrt(hb) * QMAX)


# --------------------------------------------------------------------------
# Convolution on codes (conv_ref.c) and the requantize epilogue
# --------------------------------------------------------------------------

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None


def build_lib(force: bool = False) -> str:
    out_dir = os.path.join(_HERE, "_build")
    so = os.path.join(out_dir, "liboracle.so")
    src = os.path.join(_HERE, "conv_ref.c")
    if force or not os.path.exists(so) or os.path.getmtime(so) < os.path.getmtime(src):
        os.makedirs(out_dir, exist_ok=True)
        tmp = so + f".tmp{os.getpid()}"
        base = ["gcc", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-o", tmp, src]
        if subprocess.run(base[:1] + ["-fopenmp"] + base[1:], capture_output=True).returncode != 0:
            subprocess.check_call(base)
        os.replace(tmp, so)
    return so


def _lib():
    global _LIB
    if _LIB is None:
        lib = ctypes.CDLL(build_lib())
        i64 = ctypes.c_int64
        p = ctypes.c_void_p
        lib.oracle_conv2d_codes.argtypes = [p, i64, i64, i64, i64, p, i64, i64, i64, i64, i64,
                                            i64, i64, i64, i64, p]
        lib.oracle_conv2d_codes_at.argtypes = [p, i64, i64, i64, i64, p, i64, i64, i64, i64, i64,
                                               p, i64, p]
        lib.oracle_max_threads.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        _LIB = lib
    return _LIB


def max_threads() -> int:
    """Threads the direct convolution uses (OpenMP; 1 without it)."""
    return int(_lib().oracle_max_threads())


def set_threads(t: int) -> None:
    _lib().oracle_set_threads(int(t))


def out_hw(h, w, k, stride, pad):
    return (h + 2 * pad - k) // stride + 1, (w + 2 * pad - k) // stride + 1


def conv_codes(x_i8, w_int, stride: int, pad: int, window=None) -> np.ndarray:
    """Integer accumulator sum_k x_int w_int over the unfolded patch
    (Eqs. integer_accumulation, linear_operator). x: NHWC int8, w: OHWI int8.
    window = (ho0, ho1, wo0, wo1) restricts the output rows/columns."""
    x = np.ascontiguousarray(x_i8, dtype=np.int8)
    w = np.ascontiguousarray(w_int, dtype=np.int8)
    n, h, wd, c = x.shape
    co, kh, kw, ci = w.shape
    if ci != c:
        raise ValueError("channel mismatch")
    ho, wo = out_hw(h, wd, kh, stride, pad)
    ho0, ho1, wo0, wo1 = window if window is not None else (0, ho, 0, wo)
    acc = np.zeros((n, ho1 - ho0, wo1 - wo0, co), dtype=np.int64)
    _lib().oracle_conv2d_codes(x.ctypes.data, n, h, wd, c, w.ctypes.data, co, kh, kw,
                               stride, pad, ho0, ho1, wo0, wo1, acc.ctypes.data)
    return acc


def conv_codes_at(x_i8, w_int, stride: int, pad: int, pix) -> np.ndarray:
    """The accumulator at output pixels pix[i] = (b, oy, ox): [npix, co]."""
    x = np.ascontiguousarray(x_i8, dtype=np.int8)
    w = np.ascontiguousarray(w_int, dtype=np.int8)
    pix = np.ascontiguousarray(pix, dtype=np.int64).reshape(-1, 3)
    n, h, wd, c = x.shape
    co, kh, kw, _ = w.shape
    acc = np.zeros((pix.shape[0], co), dtype=np.int64)
    _lib().oracle_conv2d_codes_at(x.ctypes.data, n, h, wd, c, w.ctypes.data, co, kh, kw,
                                  stride, pad, pix.ctypes.data, pix.shape[0], acc.ctypes.data)
    return acc


def epilogue_int(acc, p: Prepared) -> np.ndarray:
    """Integer transition of Eq. (integer_hadamard_transition) with the bias of
    Eq. (supp_bias_quantization) added first (R5):
        a = acc + b_int;  v = H~_out (M (.) a);  u = phi(v);
        x_next = clamp(round(H~_in,next(u) / 2^n), -127, 127)."""
    a = np.asarray(acc, dtype=np.int64) + p.b_int
    t = p.M * a
    v = transform_int(t, p.hb_out) if p.hb_out else t
    u = np.maximum(v, 0) if p.act == "relu" else v
    w = transform_int(u, p.hb_next) if p.hb_next else u
    return np.clip(rshift_rne(w, p.n), -QMAX, QMAX).astype(np.int8)


def epilogue_general(acc, p: Prepared) -> np.ndarray:
    """Transition through a non-homogeneous activation (Sec. general
    nonlinearities), in the order of Eqs. (supp_general_preactivation,
    supp_general_activation, supp_general_input_transition):
        z = clamp(round(H~_out (M_out (.) a) / 2^n_out)),  u = phi_int(z),
        x_next = clamp(round(H~_in,next(M_in u) / 2^n_in))."""
    a = np.asarray(acc, dtype=np.int64) + p.b_int
    t = p.M * a
    v = transform_int(t, p.hb_out) if p.hb_out else t
    z = np.clip(rshift_rne(v, p.n), -QMAX, QMAX)
    u = p.lut[z + QMAX]
    w = p.M_in * u
    w = transform_int(w, p.hb_next) if p.hb_next else w
    return np.clip(rshift_rne(w, p.n_in), -QMAX, QMAX).astype(np.int8)


def gdn(v, beta, gamma, inverse: bool = False) -> np.ndarray:
    """Generalized divisive normalization across channels (last axis), fp64:
    y_i = v_i / sqrt(beta_i + sum_j gamma_ij v_j^2); the inverse (IGDN)
    multiplies by the same root."""
    v = np.asarray(v, dtype=np.float64)
    norm = np.sqrt(np.asarray(beta, np.float64) + (v * v) @ np.asarray(gamma, np.float64).T)
    return v * norm if inverse else v / norm


class GdnParams:
    """Integer parameters of phi_int for GDN / IGDN (reading R21)."""

    def __init__(self, **kw):
        self.__dict__.update(kw)


GDN_G_MAX = 511                 # 9-bit G: G z^2 limb products stay exact in fp32 sums
GDN_D_LIMIT = 2 ** 31
GDN_P_MIN = 2 ** 15


def gdn_params(beta, gamma, s_z: float, s_u: float, inverse: bool = False) -> GdnParams:
    """phi_int of Eq. (supp_general_activation) for y_i = v_i / sqrt(beta_i +
    sum_j gamma_ij v_j^2) (IGDN: times the root) with v = s_z z, read as R21:
    the normalization pool in integers D_i = B_i + sum_j G_ij z_j^2 and the
    rounding of R |z| / sqrt(D) (IGDN: R |z| sqrt(D)) decided by squares."""
    beta = np.asarray(beta, dtype=np.float64).ravel()
    gamma = np.asarray(gamma, dtype=np.float64)
    c = beta.size
    if gamma.shape != (c, c):
        raise ValueError("gamma must be C x C")
    if not (np.all(np.isfinite(beta)) and np.all(np.isfinite(gamma))):
        raise ValueError("beta and gamma must be finite")
    if np.any(beta <= 0) or np.any(gamma < 0):
        raise ValueError("GDN needs beta > 0 and gamma >= 0")
    s_z = float(np.float32(s_z))
    s_u = float(np.float32(s_u))
    if not (s_z > 0 and s_u > 0):
        raise ValueError("scales must be positive")
    gs = gamma * s_z * s_z
    for e in range(62, -126, -1):
        if gs.max(initial=0.0) * 2.0 ** e >= GDN_G_MAX + 0.5 or beta.max() * 2.0 ** e >= GDN_D_LIMIT:
            continue
        G = np.rint(gs * 2.0 ** e).astype(np.int64)
        B = np.maximum(1, np.rint(beta * 2.0 ** e)).astype(np.int64)
        d_max = int(np.max(B + QMAX * QMAX * G.sum(axis=1)))
        if d_max < GDN_D_LIMIT:
            break
    else:
        raise OverflowError("no scaling keeps the GDN pool in range")
    r2 = (s_z / s_u) ** 2 * (2.0 ** -e if inverse else 2.0 ** e)
    for t in range(62, -1, -1):
        P = int(np.rint(math.ldexp(r2, t)))
        if inverse:
            ok = (2 * QMAX - 1) ** 2 * 2 ** t < 2 ** 63 and 4 * P * QMAX * QMAX * d_max < 2 ** 63
        else:
            ok = (2 * QMAX - 1) ** 2 * d_max * 2 ** t < 2 ** 63 and 4 * P * QMAX * QMAX < 2 ** 63
        if ok:
            break
    else:
        raise OverflowError("no fixed-point R^2 fits the 63-bit tests")
    if P < GDN_P_MIN:
        raise OverflowError("fewer than 16 bits in the fixed-point R^2")
    return GdnParams(G=G, B=B, e=e, P=P, t=t, inverse=bool(inverse), d_max=d_max, c=c)


def gdn_pool(z, g: GdnParams) -> np.ndarray:
    """D_i = B_i + sum_j G_ij z_j^2 over the last axis (exact int64)."""
    z2 = np.asarray(z, dtype=np.int64) ** 2
    return g.B + z2 @ g.G.T


def isqrt_floor(q) -> np.ndarray:
    """floor(sqrt(q)) elementwise for 0 <= q < 2^52, exact (float estimate
    corrected by integer comparisons)."""
    q = np.asarray(q, dtype=np.int64)
    s = np.floor(np.sqrt(q.astype(np.float64))).astype(np.int64)
    s = np.where(s * s > q, s - 1, s)
    s = np.where((s + 1) * (s + 1) <= q, s + 1, s)
    return s


def gdn_int(z, g: GdnParams) -> np.ndarray:
    """u = phi_int(z) for GDN / IGDN (R21): |u| is the largest k <= 127 with
    (2k - 1)^2 Den <= Num, i.e. k <= (isqrt(floor(Num / Den)) + 1) / 2, where
    GDN: Num = 4 P z^2, Den = D 2^t; IGDN: Num = 4 P z^2 D, Den = 2^t."""
    z = np.asarray(z, dtype=np.int64)
    D = gdn_pool(z, g)
    z2 = z * z
    if g.inverse:
        q = (4 * g.P * z2 * D) >> g.t
    else:
        q = (4 * g.P * z2) // (D << g.t)
    q = np.minimum(q, (2 * QMAX + 1) ** 2)        # any S >= 253 gives |u| = 127
    k = np.minimum(QMAX, (isqrt_floor(q) + 1) // 2)
    return np.sign(z) * k


def input_transition(u, p: Prepared) -> np.ndarray:
    """Eq. (supp_general_input_transition): x_next = clamp(round(H~_in,next
    (M_in u) / 2^n_in), -127, 127)."""
    w = p.M_in * np.asarray(u, dtype=np.int64)
    w = transform_int(w, p.hb_next) if p.hb_next else w
    return np.clip(rshift_rne(w, p.n_in), -QMAX, QMAX).astype(np.int8)


def preactivation(acc, p: Prepared) -> np.ndarray:
    """Eq. (supp_general_preactivation): z = clamp(round(H~_out (M_out (.) a)
    / 2^n_out), -127, 127) with a = acc + b_int."""
    a = np.asarray(acc, dtype=np.int64) + p.b_int
    t = p.M * a
    v = transform_int(t, p.hb_out) if p.hb_out else t
    return np.clip(rshift_rne(v, p.n), -QMAX, QMAX)


def epilogue_general_vector(acc, p: Prepared) -> np.ndarray:
    """The transition of Sec. general nonlinearities for a channel-coupled
    activation (GDN / IGDN): z by Eq. supp_general_preactivation, u = phi_int(z)
    on each pixel's channel vector (R21), then the input-side rescale."""
    return input_transition(gdn_int(preactivation(acc, p), p.gdn), p)


def epilogue_f32(acc, p: Prepared) -> np.ndarray:
    """Dequantized output: y = H_out (s_A (.) a) (WH) or s_A (.) a (DH), then phi;
    with deq_c = s_x s_w,c / gamma_out the WH form is H~_out (deq (.) a)."""
    a = np.asarray(acc, dtype=np.int64) + p.b_int
    t = p.deq * a.astype(np.float64)
    v = transform_real(t, p.hb_out, normalize=False) if p.hb_out else t
    return np.maximum(v, 0.0) if p.act == "relu" else v


def conv_layer(x_op, p: Prepared, window=None):
    """One prepared layer on its INT8 operand: conv + epilogue."""
    acc = conv_codes(x_op, p.w_int, p.stride, p.pad, window)
    if p.act in GENERAL_ACTS:
        return epilogue_general(acc, p)
    return epilogue_f32(acc, p) if p.out_f32 else epilogue_int(acc, p)


# --------------------------------------------------------------------------
# Layer stacking by the static profile mask (Sec. layer-wise selection,
# Table integer_transitions)
# --------------------------------------------------------------------------


def layer_operand(x, x_kind: str, s_in: float, form: str, hb_in: int, s_x: float):
    """The INT8 operand a layer consumes from its input.
    x_kind: 'operand' (already the operand), 'i8' (original-basis codes at
    s_in) or 'f16' (real values). DH applies the input transform (hb_in);
    WH only rescales (identity transform)."""
    hb = hb_in if form == "DH" else 1
    if x_kind == "operand":
        return np.asarray(x, dtype=np.int8)
    if x_kind == "f16":
        return quantize_act_f16(x, hb, s_x)
    if x_kind == "i8":
        if form == "WH" and float(np.float32(s_in)) == float(np.float32(s_x)):
            return np.asarray(x, dtype=np.int8)
        return quantize_act_i8(x, hb, s_in, s_x)
    raise ValueError(x_kind)


def transition_blocks(layers):
    """Per layer l, the block of the input-side transform H~_in,l+1 that layer
    l's transition applies after phi (Table integer_transitions): the next
    layer's input block when it is DH (DH-to-DH, WH-to-DH), 0 when it is WH
    or there is none (DH-to-WH, WH-to-WH, last layer). Every transition inside
    a chain is one requantization with one round-shift
    (Eq. integer_hadamard_transition), whatever the blocks are."""
    out = []
    for i in range(len(layers)):
        nxt = layers[i + 1] if i + 1 < len(layers) else None
        out.append(nxt.hb_in if nxt is not None and nxt.form == "DH" else 0)
    return out


def prepare_chain(layers, params, scales, out_f32_last=False):
    """layers: LayerSpec-like objects; params: [(w, b)]; scales: [{'s_x','s_out'}]
    (s_out: the scale of the next layer's operand, or of the chain output).
    Each layer is prepared with the input-side block of its transition."""
    hb_next = transition_blocks(layers)
    preps = []
    for i, (L, (w, b), sc) in enumerate(zip(layers, params, scales)):
        last = i == len(layers) - 1
        preps.append(prepare_layer(w, b, L.form, L.hb_in, L.hb_out, sc["s_x"], sc["s_out"],
                                   L.act, hb_next[i], out_f32_last and last, L.stride, L.pad))
    return preps


def chain_forward(layers, preps, x, x_kind, s_in):
    """Run a chain on the oracle. The chain input enters its first layer through
    layer_operand; every later layer consumes its producer's output as is (the
    producer's transition already emitted the operand in the consumer's basis
    and scale). Returns the list of per-layer outputs."""
    outs = []
    cur, kind, s_cur = x, x_kind, s_in
    for L, p in zip(layers, preps):
        op = layer_operand(cur, kind, s_cur, L.form, L.hb_in, p.s_x)
        y = conv_layer(op, p)
        outs.append(y)
        cur, kind, s_cur = y, "operand", p.s_y
    return outs


# --------------------------------------------------------------------------
# Real-valued model (fp64): the function the quantized operator approximates
# --------------------------------------------------------------------------


def conv_real(x, w_ohwi, b, stride: int, pad: int) -> np.ndarray:
    """Y = X W^T + b on unfolded patches (Eq. supp_linear_operator), fp64,
    with a library matmul per kernel tap."""
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w_ohwi, dtype=np.float64)
    n, h, wd, c = x.shape
    co, kh, kw, _ = w.shape
    ho, wo = out_hw(h, wd, kh, stride, pad)
    xp = np.zeros((n, h + 2 * pad, wd + 2 * pad, c))
    xp[:, pad:pad + h, pad:pad + wd, :] = x
    y = np.zeros((n, ho, wo, co))
    for ky in range(kh):
        for kx in range(kw):
            patch = xp[:, ky:ky + stride * (ho - 1) + 1:stride, kx:kx + stride * (wo - 1) + 1:stride, :]
            y += patch @ w[:, ky, kx, :].T
    if b is not None:
        y += np.asarray(b, dtype=np.float64)
    return y


# --------------------------------------------------------------------------
# Dynamic affine activation quantization (PTQ setting): Eqs. (uniform_q,
# affine_q); the MACs and transforms use centred codes x_int - z_x
# (supplementary, affine activation quantization)
# --------------------------------------------------------------------------

AFFINE_QMIN, AFFINE_QMAX = 0, 255          # unsigned 8-bit grid of Eq. affine_q


def affine_params(x):
    """(s, z) of Eq. affine_q from the tensor's range, zero kept representable:
    x_min' = min(x_min, 0), x_max' = max(x_max, 0), s = (x_max' - x_min') / 255,
    z = clamp(round(0 - x_min' / s), 0, 255); a zero range gives (1, 0), and so
    does a range too small for a nonzero step (s underflows to 0)."""
    x = np.asarray(x, dtype=np.float64)
    lo = min(float(x.min()), 0.0) if x.size else 0.0
    hi = max(float(x.max()), 0.0) if x.size else 0.0
    if hi - lo <= 0.0:
        return 1.0, 0
    s = (hi - lo) / (AFFINE_QMAX - AFFINE_QMIN)
    if not s > 0.0:
        return 1.0, 0
    z = int(min(max(round(AFFINE_QMIN - lo / s), AFFINE_QMIN), AFFINE_QMAX))
    return s, z


def quantize_affine(x, s: float, z: int) -> np.ndarray:
    """x_int = clamp(round(x / s) + z, 0, 255) of Eq. uniform_q."""
    q = np.rint(np.asarray(x, dtype=np.float64) / s) + z
    return np.clip(q, AFFINE_QMIN, AFFINE_QMAX).astype(np.int64)


def conv_codes_wide(x_int, w_int, stride: int, pad: int) -> np.ndarray:
    """The integer accumulator for codes wider than INT8 (centred affine codes,
    |x| <= 255): a library matmul per kernel tap in int64, zero padding."""
    x = np.asarray(x_int, dtype=np.int64)
    w = np.asarray(w_int, dtype=np.int64)
    n, h, wd, c = x.shape
    co, kh, kw, _ = w.shape
    ho, wo = out_hw(h, wd, kh, stride, pad)
    xp = np.zeros((n, h + 2 * pad, wd + 2 * pad, c), dtype=np.int64)
    xp[:, pad:pad + h, pad:pad + wd, :] = x
    acc = np.zeros((n, ho, wo, co), dtype=np.int64)
    for ky in range(kh):
        for kx in range(kw):
            patch = xp[:, ky:ky + stride * (ho - 1) + 1:stride, kx:kx + stride * (wo - 1) + 1:stride, :]
            acc += patch @ w[:, ky, kx, :].T
    return acc


def conv_layer_affine(x_real, p: Prepared):
    """A prepared layer (out_f32 preparation: DH / WH weights, s_w, bias) on a
    real input with dynamic affine activation quantization: the input-side
    operand (T x for DH, x for WH) is quantized with (s, z) from its own range,
    the convolution runs on the centred codes x_int - z (zero padding is a
    centred zero), and the output is dequantized:
    y = H_out(s s_w (.) a) + b_bar, a = sum (x_int - z) w_int.
    Returns (y, s, z)."""
    v = transform_real(np.asarray(x_real, dtype=np.float64), p.hb_in) if p.form == "DH" else \
        np.asarray(x_real, dtype=np.float64)
    s, z = affine_params(v)
    centred = quantize_affine(v, s, z) - z
    return conv_layer_affine_codes(centred, s, p), s, z


def conv_layer_affine_codes(centred, s: float, p: Prepared):
    """The second half of conv_layer_affine: the convolution on centred codes
    at step s and the dequantized output y = phi(H_out(s s_w (.) a) + b_bar)."""
    acc = conv_codes_wide(centred, p.w_int, p.stride, p.pad)
    t = (s * p.s_w) * acc.astype(np.float64)
    y = transform_real(t, p.hb_out) if p.form == "WH" else t
    y = y + p.bbar if p.form == "DH" else y + transform_real(p.bbar, p.hb_out)
    return np.maximum(y, 0.0) if p.act == "relu" else y


# --------------------------------------------------------------------------
# Decoder-side operators (synthesis transforms): transposed and sub-pixel
# convolutions, linear operators Y = X W^T of Eq. (linear_operator) like the
# analysis convolutions, so the DH / WH weight transforms apply unchanged
# (DH along the contracted C_in, WH along C_out).
# --------------------------------------------------------------------------


def conv_transpose_hw(h, w, k, stride, pad, out_pad=0):
    return (h - 1) * stride - 2 * pad + k + out_pad, (w - 1) * stride - 2 * pad + k + out_pad


def conv_transpose_real(x, w_ohwi, b, stride: int, pad: int, out_pad: int = 0) -> np.ndarray:
    """Transposed convolution, fp64: every input pixel (iy, ix) scatters
    x[iy, ix, :] W[:, ky, kx, :]^T to output pixel (iy s + ky - pad, ix s + kx - pad).
    w_ohwi: [C_out, kh, kw, C_in] of this layer (C_in -> C_out)."""
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w_ohwi, dtype=np.float64)
    n, h, wd, c = x.shape
    co, kh, kw, _ = w.shape
    ho, wo = conv_transpose_hw(h, wd, kh, stride, pad, out_pad)
    big = np.zeros((n, (h - 1) * stride + kh, (wd - 1) * stride + kw, co))
    for ky in range(kh):
        for kx in range(kw):
            big[:, ky:ky + stride * (h - 1) + 1:stride, kx:kx + stride * (wd - 1) + 1:stride, :] += x @ w[:, ky, kx, :].T
    y = np.zeros((n, ho, wo, co))
    hh, ww = min(ho, big.shape[1] - pad), min(wo, big.shape[2] - pad)
    y[:, :hh, :ww, :] = big[:, pad:pad + hh, pad:pad + ww, :]
    if b is not None:
        y += np.asarray(b, dtype=np.float64)
    return y


def conv_transpose_codes(x_i8, w_int, stride: int, pad: int, out_pad: int = 0) -> np.ndarray:
    """The same scatter on INT8 codes, exact in int64."""
    x = np.asarray(x_i8, dtype=np.int64)
    w = np.asarray(w_int, dtype=np.int64)
    n, h, wd, c = x.shape
    co, kh, kw, _ = w.shape
    ho, wo = conv_transpose_hw(h, wd, kh, stride, pad, out_pad)
    big = np.zeros((n, (h - 1) * stride + kh, (wd - 1) * stride + kw, co), dtype=np.int64)
    for ky in range(kh):
        for kx in range(kw):
            big[:, ky:ky + stride * (h - 1) + 1:stride, kx:kx + stride * (wd - 1) + 1:stride, :] += x @ w[:, ky, kx, :].T
    y = np.zeros((n, ho, wo, co), dtype=np.int64)
    hh, ww = min(ho, big.shape[1] - pad), min(wo, big.shape[2] - pad)
    y[:, :hh, :ww, :] = big[:, pad:pad + hh, pad:pad + ww, :]
    return y


def conv_transpose_layer(x_op, p: Prepared, out_pad: int = 0):
    """A prepared layer (prepare_layer: DH / WH weights, bias codes, (M, n))
    applied as a transposed convolution, then the integer transition."""
    acc = conv_transpose_codes(x_op, p.w_int, p.stride, p.pad, out_pad)
    if p.act in GENERAL_ACTS:
        return epilogue_general(acc, p)
    return epilogue_f32(acc, p) if p.out_f32 else epilogue_int(acc, p)


def depth_to_space(x, r: int) -> np.ndarray:
    """Sub-pixel rearrangement: NHWC [n, h, w, c r^2] -> [n, h r, w r, c], channel
    c r^2 + i r + j going to pixel (h r + i, w r + j), channel c."""
    x = np.asarray(x)
    n, h, w, crr = x.shape
    if crr % (r * r):
        raise ValueError("channels must be a multiple of r^2")
    c = crr // (r * r)
    return x.reshape(n, h, w, c, r, r).transpose(0, 1, 4, 2, 5, 3).reshape(n, h * r, w * r, c)


def space_to_depth(x, r: int) -> np.ndarray:
    """Inverse of depth_to_space."""
    x = np.asarray(x)
    n, hr, wr, c = x.shape
    h, w = hr // r, wr // r
    return x.reshape(n, h, r, w, r, c).transpose(0, 1, 3, 5, 2, 4).reshape(n, h, w, c * r * r)


def calibrate_chain(layers, params, x_real, first_wh_scale=None):
    """Static scales from the real-valued model (QAT-style frozen scales,
    Sec. quantization-aware training): per layer, s_x = max-abs of the
    operand in its quantizer's basis / 127, and s_out = the scale of what the
    layer emits: the next layer's operand (in the next layer's input basis,
    i.e. after H_in,l+1 when the next layer is DH), or the chain output."""
    scales = []
    x = np.asarray(x_real, dtype=np.float64)
    reals = []
    for i, (L, (w, b)) in enumerate(zip(layers, params)):
        if L.form == "DH":
            s_x = symmetric_scale(transform_real(x, L.hb_in))
        else:
            s_x = symmetric_scale(x) if (i or first_wh_scale is None) else first_wh_scale
        y = conv_real(x, w, b, L.stride, L.pad)
        xn = np.maximum(y, 0.0) if L.act == "relu" else y
        reals.append((x, xn))
        scales.append({"s_x": float(np.float32(s_x))})
        x = xn
    hb_next = transition_blocks(layers)
    for i, L in enumerate(layers):
        xn = reals[i][1]
        if hb_next[i]:
            s_out = symmetric_scale(transform_real(xn, hb_next[i]))
        else:
            s_out = symmetric_scale(xn)
        scales[i]["s_out"] = float(np.float32(s_out))
    return scales


# --------------------------------------------------------------------------
# Diagnostics: Eqs. (excess_kurtosis, sqnr, hadamard_sensitivity)
# --------------------------------------------------------------------------


def excess_kurtosis(x) -> float:
    x = np.asarray(x, dtype=np.float64).ravel()
    mu = x.mean()
    d = x - mu
    return float(np.mean(d ** 4) / np.mean(d ** 2) ** 2 - 3.0)


def sqnr_db(x, xhat) -> float:
    x = np.asarray(x, dtype=np.float64)
    e = x - np.asarray(xhat, dtype=np.float64)
    return float(10.0 * np.log10(np.sum(x * x) / np.sum(e * e)))


def range_expands(x, hb: int) -> bool:
    """Indicator of Eq. (hadamard_sensitivity) for one tensor."""
    return float(np.max(np.abs(transform_real(x, hb)))) > float(np.max(np.abs(x)))


# --------------------------------------------------------------------------
# Profiling-based strategy selection: Eqs. (hadamard_sensitivity,
# layerwise_hadamard_selection), on the INT8 codes a layer receives
# --------------------------------------------------------------------------


def range_expansion_codes(x_i8, hb: int):
    """Per image k of an NHWC code tensor, the indicator of Eq.
    (hadamard_sensitivity), ||T x_k||_inf > ||x_k||_inf with the normalized
    block transform T = I (x) H~_hb / sqrt(hb). With integer codes it is decided
    exactly as max|H~_hb x_k|^2 > hb * max|x_k|^2 (Python integers).
    Returns (max|x_k|, max|H~ x_k|, indicator) as int64, int64, uint8 arrays."""
    x = np.asarray(x_i8, dtype=np.int64)
    n = x.shape[0]
    flat = x.reshape(n, -1, x.shape[-1])
    y = transform_int(flat, hb)
    mx = np.abs(flat).reshape(n, -1).max(axis=1) if flat.size else np.zeros(n, np.int64)
    mh = np.abs(y).reshape(n, -1).max(axis=1) if y.size else np.zeros(n, np.int64)
    ind = np.array([int(h) ** 2 > hb * int(m) ** 2 for h, m in zip(mh, mx)], dtype=np.uint8)
    return mx.astype(np.int64), mh.astype(np.int64), ind


def expansion_probability(indicators) -> Fraction:
    """p_l of Eq. (hadamard_sensitivity): the fraction of the M profiled images
    whose range expands, as an exact rational."""
    ind = [int(v) for v in np.asarray(indicators).ravel()]
    if not ind:
        raise ValueError("no profiled images")
    return Fraction(sum(ind), len(ind))


def select_form(p, tau=Fraction(4, 5)) -> str:
    """pi_l of Eq. (layerwise_hadamard_selection): WH when p_l > tau_sel, else
    DH (the paper uses tau_sel = 0.8)."""
    return "WH" if Fraction(p) > Fraction(tau) else "DH"
