"""Test helpers that hold none of the method's arithmetic: fixture loading and comparisons."""
import json
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def pack_rollouts(rollouts):
    """List of token lists -> (ids int32, off int64)."""
    lens = [len(r) for r in rollouts]
    off = np.zeros(len(rollouts) + 1, np.int64)
    off[1:] = np.cumsum(lens)
    ids = np.array([t for r in rollouts for t in r], np.int32) if off[-1] else np.zeros(0, np.int32)
    return ids, off


def bf16_ordered(bits):
    """bf16 bit patterns (uint16) -> integers ordered like the values (+0 and -0 both 0)."""
    b = np.asarray(bits).astype(np.int32)
    neg = (b & 0x8000) != 0
    mag = b & 0x7FFF
    return np.where(neg, -mag, mag)


def bf16_ulp_distance(a_bits, b_bits):
    return np.abs(bf16_ordered(a_bits) - bf16_ordered(b_bits))


def bf16_bits_to_f32(bits):
    return (np.asarray(bits).astype(np.uint32) << 16).view(np.float32)
