"""Counter-based synthetic data: SplitMix64 streams, Irwin-Hall-12 normals, BF16.

Definition (the same text is the contract for the CUDA and C implementations):

* ``mix64(z)`` is the SplitMix64 output finalizer of Steele, Lea and Flood
  (OOPSLA 2014, "Fast splittable pseudorandom number generators"), with the
  multipliers 0xBF58476D1CE4E5B9 / 0x94D049BB133111EB and shifts 30/27/31, all
  arithmetic modulo 2**64.
* SplitMix64 started at state ``key`` returns, as its n-th output (n = 0, 1, ...),
  ``draw(key, n) = mix64(key + (n + 1) * GOLDEN)`` with GOLDEN = 0x9E3779B97F4A7C15.
  Because the state advances by a constant, any output is reachable by index.
* ``stream_key(seed, tensor, layer, sub)`` folds four 64-bit words with
  ``h(z) = mix64(z + GOLDEN)``: ``h(h(h(h(seed) ^ tensor) ^ layer) ^ sub)``.
* ``normal(key, i)``: the twelve 16-bit lanes of draws 3i, 3i+1, 3i+2 are summed
  (lane order is irrelevant to the sum) into an integer S in [0, 12*65535]; the
  value is ``(S - 393210) * 2**-16`` which is exact in FP32 (|S-393210| < 2**20).
  Mean 0, variance (65536**2-1)/65536**2, support [-6, 6].
* A tensor of standard deviation sigma holds ``fl32(normal * fl32(sigma))`` (one
  IEEE single-precision multiply, no fused operation).
* BF16 tensors hold the FP32 value rounded to nearest-even in the top 16 bits.
* Element index of a row-major [rows, cols] tensor is ``row * cols + col``.
"""
from __future__ import annotations

import numpy as np

GOLDEN = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1
LANE_MEAN_SUM = 393210  # 12 lanes * 65535 / 2

# Tensor ids of the synthetic model and its inputs.
T_WQ = 1
T_WK = 2
T_WV = 3
T_WO = 4
T_WGATE = 5
T_WUP = 6
T_WDOWN = 7
T_GAMMA_ATTN = 8
T_GAMMA_MLP = 9
T_GAMMA_FINAL = 10
T_LMHEAD = 11
T_KCACHE = 20
T_VCACHE = 21
T_XSTEP = 30
T_PROMPT = 31
T_SCORE = 40
T_TARGET = 41
T_TURN = 42
T_PROBE = 50

WEIGHT_SIGMA = 0.02
GAMMA_SIGMA = 0.02

_U64 = np.uint64


def mix64_int(z: int) -> int:
    """SplitMix64 finalizer on a Python int (mod 2**64)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 finalizer on a uint64 array (in place on a private copy)."""
    z = np.array(z, dtype=_U64, copy=True)
    z ^= z >> _U64(30)
    z *= _U64(MIX1)
    z ^= z >> _U64(27)
    z *= _U64(MIX2)
    z ^= z >> _U64(31)
    return z


def _h(z: int) -> int:
    return mix64_int((z + GOLDEN) & MASK64)


def stream_key(seed: int, tensor: int, layer: int = 0, sub: int = 0) -> int:
    """64-bit key of the stream for (seed, tensor id, layer, sub-index)."""
    k = _h(seed & MASK64)
    k = _h(k ^ (tensor & MASK64))
    k = _h(k ^ (layer & MASK64))
    k = _h(k ^ (sub & MASK64))
    return k


def splitmix64_sequence(seed: int, count: int) -> list[int]:
    """The first ``count`` outputs of a SplitMix64 generator whose state is ``seed``."""
    return [mix64_int(seed + (n + 1) * GOLDEN) for n in range(count)]


def draws(key: int, n: np.ndarray) -> np.ndarray:
    """Outputs number ``n`` (uint64 array of indices) of the stream ``key``."""
    n = np.asarray(n, dtype=_U64)
    with np.errstate(over="ignore"):
        state = _U64(key) + (n + _U64(1)) * _U64(GOLDEN)
    return mix64(state)


def normal_at(key: int, idx: np.ndarray) -> np.ndarray:
    """Irwin-Hall-12 normals (float32) at element indices ``idx``."""
    idx = np.asarray(idx, dtype=_U64)
    s = np.zeros(idx.shape, dtype=np.int64)
    for k in range(3):
        d = draws(key, idx * _U64(3) + _U64(k))
        for j in range(4):
            s += ((d >> _U64(16 * j)) & _U64(0xFFFF)).astype(np.int64)
    return (s - LANE_MEAN_SUM).astype(np.float32) * np.float32(1.0 / 65536.0)


def normal_range(key: int, start: int, count: int) -> np.ndarray:
    """Irwin-Hall-12 normals for element indices start .. start+count-1."""
    return normal_at(key, np.arange(start, start + count, dtype=_U64))


def scaled(z: np.ndarray, sigma: float) -> np.ndarray:
    """fl32(z * fl32(sigma)): one IEEE single multiply."""
    return (z.astype(np.float32) * np.float32(sigma)).astype(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to BF16 (nearest-even) and return the uint16 bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (b + _U64(0x7FFF) + ((b >> _U64(16)) & _U64(1))) >> _U64(16)
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen BF16 bit patterns (uint16) to float32 values (exact)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """float32 values rounded to the nearest BF16 value (returned as float32)."""
    return bf16_to_f32(bf16_bits(x))


def uniform_u32(key: int, idx: np.ndarray) -> np.ndarray:
    """High 32 bits of draw ``idx``: uniform integers in [0, 2**32)."""
    return (draws(key, idx) >> _U64(32)).astype(np.uint32)


def uniform_u24(key: int, idx: np.ndarray) -> np.ndarray:
    """High 24 bits of draw ``idx``: uniform integers in [0, 2**24)."""
    return (draws(key, idx) >> _U64(40)).astype(np.uint32)


# ---------------------------------------------------------------------------
# Keyed recipes of the synthetic workload.
# ---------------------------------------------------------------------------

def weight_f32(seed: int, tensor: int, layer: int, rows: int, cols: int,
               row0: int = 0, nrows: int | None = None) -> np.ndarray:
    """Dense FP32 weight rows [row0, row0+nrows) of a [rows, cols] matrix, N(0, 0.02)."""
    if nrows is None:
        nrows = rows - row0
    key = stream_key(seed, tensor, layer, 0)
    z = normal_range(key, row0 * cols, nrows * cols).reshape(nrows, cols)
    return scaled(z, WEIGHT_SIGMA)


def gamma_f32(seed: int, tensor: int, layer: int, d: int) -> np.ndarray:
    """RMSNorm gain 1 + N(0, 0.02), as fl32(1 + fl32(z * 0.02))."""
    key = stream_key(seed, tensor, layer, 0)
    z = scaled(normal_range(key, 0, d), GAMMA_SIGMA)
    return (np.float32(1.0) + z).astype(np.float32)


def lm_head_bf16(seed: int, vocab: int, d: int, row0: int = 0,
                 nrows: int | None = None) -> np.ndarray:
    """BF16 bit patterns of LM-head rows [row0, row0+nrows), N(0, 0.02)."""
    if nrows is None:
        nrows = vocab - row0
    key = stream_key(seed, T_LMHEAD, 0, 0)
    z = normal_range(key, row0 * d, nrows * d).reshape(nrows, d)
    return bf16_bits(scaled(z, WEIGHT_SIGMA))


def kv_prior_bf16(kv_seed: int, layer: int, group: int, t_prior: int, dh: int,
                  which: int) -> np.ndarray:
    """BF16 bits of a prior K (which=T_KCACHE) or V (T_VCACHE) cache block [t_prior, dh], N(0,1)."""
    key = stream_key(kv_seed, which, layer, group)
    return bf16_bits(normal_range(key, 0, t_prior * dh)).reshape(t_prior, dh)


def step_inputs_bf16(seed: int, n_steps: int, n: int, d: int, session0: int = 0) -> np.ndarray:
    """BF16 bits of teacher-forced decode inputs x_t, shape [n_steps, n, d], N(0,1)."""
    out = np.empty((n_steps, n, d), dtype=np.uint16)
    for t in range(n_steps):
        for s in range(n):
            key = stream_key(seed, T_XSTEP, t, session0 + s)
            out[t, s] = bf16_bits(normal_range(key, 0, d))
    return out


def prompt_bf16(seed: int, turn: int, T: int, d: int) -> np.ndarray:
    """BF16 bits of a synthetic prompt's embeddings [T, d], N(0,1)."""
    key = stream_key(seed, T_PROMPT, turn, 0)
    return bf16_bits(normal_range(key, 0, T * d)).reshape(T, d)


def probe_f32(seed: int, tag: int, d: int, sigma: float = 1.0) -> np.ndarray:
    """An FP32 probe vector N(0, sigma^2) (e.g. an isolated layer's input residual)."""
    key = stream_key(seed, T_PROBE, tag, 0)
    return scaled(normal_range(key, 0, d), sigma)


def mask_scores_u32(mask_seed: int, L: int, n_units: int) -> np.ndarray:
    """Stand-in sensitivity scores s_h (uint32) [L, n_units]; units = groups then channel units."""
    out = np.empty((L, n_units), dtype=np.uint32)
    for layer in range(L):
        key = stream_key(mask_seed, T_SCORE, layer, 0)
        out[layer] = uniform_u32(key, np.arange(n_units, dtype=_U64))
    return out


def layer_target_u24(mask_seed: int, L: int) -> np.ndarray:
    """Per-layer retention draws (uint32 in [0, 2**24)), one per layer."""
    key = stream_key(mask_seed, T_TARGET, 0, 0)
    return uniform_u24(key, np.arange(L, dtype=_U64))


def turn_assignment(seed: int, n_turns: int, n_masks: int, p_dense: float,
                    len_lo: int, len_hi: int) -> list[tuple[int, int]]:
    """Mixed-turn serving draws: per turn (plan index, prompt length).

    Plan index ``n_masks`` denotes the dense fallback (taken with probability
    ``p_dense``); otherwise one of the masks uniformly. Prompt lengths are
    uniform integers in [len_lo, len_hi].
    """
    key = stream_key(seed, T_TURN, 0, 0)
    out = []
    for t in range(n_turns):
        d = draws(key, np.array([3 * t, 3 * t + 1, 3 * t + 2], dtype=_U64))
        u_dense = int(d[0] >> _U64(40)) / float(1 << 24)
        if u_dense < p_dense:
            plan = n_masks
        else:
            plan = int(d[1] >> _U64(32)) % n_masks
        length = len_lo + int(d[2] >> _U64(32)) % (len_hi - len_lo + 1)
        out.append((plan, length))
    return out
