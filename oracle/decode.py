"""Oracle for decode attention over the compressed cache, in float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Sec. 2 ("VLLM Decoding"): every decode step's query attends to the cached
keys and values; after PruneKV (Sec. 3.2) the visual part of layer l's cache
is the compressed (K_new, V_new) of B_l rows per KV head, so the step reads
B_l visual rows instead of n.  Here, for one layer:

    out_j = softmax(q_j K_g^T * scale) V_g,   g = j // G,

over the concatenation of the layer's kept visual rows and the text rows of
KV head g, scale 1/sqrt(d) (scaled dot-product attention).  Readings: a
query with no keys at all (an evicted layer without text) returns zeros.
"""
from __future__ import annotations

from typing import Optional

import numpy as np


def decode_attention(q: np.ndarray, K_vis: np.ndarray, V_vis: np.ndarray,
                     K_text: Optional[np.ndarray] = None, V_text: Optional[np.ndarray] = None,
                     scale: Optional[float] = None) -> np.ndarray:
    """q [Hq][d]; K_vis, V_vis [Hkv][B][d]; K_text, V_text [Hkv][T][d] -> out [Hq][d]."""
    q = np.asarray(q, dtype=np.float64)
    Hq, d = q.shape
    Hkv = K_vis.shape[0]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    out = np.zeros((Hq, d))
    for j in range(Hq):
        g = j // G
        Ks, Vs = [np.asarray(K_vis[g], np.float64)], [np.asarray(V_vis[g], np.float64)]
        if K_text is not None:
            Ks.append(np.asarray(K_text[g], np.float64))
            Vs.append(np.asarray(V_text[g], np.float64))
        Kc, Vc = np.concatenate(Ks), np.concatenate(Vs)
        if Kc.shape[0] == 0:
            continue
        x = (Kc @ q[j]) * scale
        p = np.exp(x - x.max())
        out[j] = (p / p.sum()) @ Vc
    return out
