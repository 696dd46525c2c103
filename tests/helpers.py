"""Shared test helpers: building workloads from explicit probability rows."""
import json
import os

import numpy as np

from paper_2405_19261_gb300.workloads import Workload, f32_to_bf16_bits

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load_golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def rows_workload(q_probs, p_probs, tokens, uniforms, rule, alpha, temperature=1.0,
                  dtype="f32", B=1):
    """A one-sequence workload (tiled B times) whose logits are log-probabilities."""
    with np.errstate(divide="ignore"):  # probability 0 is the logit -inf
        q = np.log(np.asarray(q_probs, np.float64)).astype(np.float32)
        p = np.log(np.asarray(p_probs, np.float64)).astype(np.float32)
    gamma, V = q.shape
    assert p.shape == (gamma + 1, V)
    q = np.broadcast_to(q * np.float32(temperature), (B, gamma, V)).copy()
    p = np.broadcast_to(p * np.float32(temperature), (B, gamma + 1, V)).copy()
    if dtype == "bf16":
        q, p = f32_to_bf16_bits(q), f32_to_bf16_bits(p)
    tok = np.broadcast_to(np.asarray(tokens, np.int32), (B, gamma)).copy()
    u = np.asarray(uniforms, np.float32).reshape(-1, gamma + 1)
    if u.shape[0] == 1:
        u = np.broadcast_to(u, (B, gamma + 1)).copy()
    return Workload(name="rows", B=B, gamma=gamma, V=V, dtype=dtype, draft=q, target=p,
                    tokens=tok, uniforms=u, rule=rule, alpha=float(alpha),
                    temperature=float(temperature))


def np_softmax(z, temperature):
    """Reference softmax via scipy (float64)."""
    from scipy.special import softmax
    return softmax(np.asarray(z, np.float64) / temperature, axis=-1)
