"""Oracle: the layer-group precision masks (test infrastructure).

Layer indices L = {0, ..., 25} (FFN section).  The FFN groupings are Eq. ffn55, ffn1010 and
ffnall26; the Attention + FFN configurations take Q_ATT = L (Attention section and
Eq. attnffn55, attnffn1010); lm_head is a separate switch (LM Head section).  A mask is the
triple (Q_FFN, Q_ATT, lm_head); layers outside a set keep bf16.

The bit encoding (bit l of a uint32 set when layer l is in the set) is the one the C-ABI uses.
"""
from __future__ import annotations

from typing import NamedTuple

NUM_LAYERS = 26
L = frozenset(range(NUM_LAYERS))

GROUPS = {
    "none": frozenset(),
    "5+5": frozenset(range(0, 5)) | frozenset(range(21, 26)),     # Eq. ffn55
    "10+10": frozenset(range(0, 10)) | frozenset(range(16, 26)),  # Eq. ffn1010
    "all26": L,                                                    # Eq. ffnall26
}


class Mask(NamedTuple):
    ffn: frozenset
    att: frozenset
    lm: bool

    def bits(self):
        """(ffn_bits, att_bits, lm) with bit l set for layer l."""
        return (sum(1 << l for l in self.ffn), sum(1 << l for l in self.att), int(self.lm))

    def n_int8_sublayers(self) -> int:
        return len(self.ffn) + len(self.att) + int(self.lm)


def make_mask(ffn: str = "none", att: str = "none", lm: bool = False) -> Mask:
    return Mask(GROUPS[ffn], GROUPS[att], bool(lm))


# The 13 configurations of the Combined Configurations table plus the fp16 (here bf16)
# baseline, named as in the table.
PAPER_CONFIGS = {
    "FP16 baseline": make_mask(),
    "attn_ffn 5+5": make_mask("5+5", "all26"),
    "FFN 5+5": make_mask("5+5"),
    "attn_ffn all26": make_mask("all26", "all26"),
    "attn_ffn 10+10": make_mask("10+10", "all26"),
    "lm_head only": make_mask(lm=True),
    "FFN 10+10": make_mask("10+10"),
    "FFN all26": make_mask("all26"),
    "attn_ffn 5+5 + lm_head": make_mask("5+5", "all26", True),
    "FFN 5+5 + lm_head": make_mask("5+5", lm=True),
    "attn_ffn 10+10 + lm_head": make_mask("10+10", "all26", True),
    "FFN 10+10 + lm_head": make_mask("10+10", lm=True),
    "Full INT8 (attn_ffn all26 + lm_head)": make_mask("all26", "all26", True),
    "FFN all26 + lm_head": make_mask("all26", lm=True),
}


def candidate_masks():
    """The sweep's candidate set: Q_FFN in {none, 5+5, 10+10, all26} x Q_ATT in {none, all26}
    x lm_head in {off, on} = 16 masks (the paper's 13 + baseline, plus attention-only with and
    without lm_head).  Returned as an ordered dict name -> Mask."""
    out = {}
    for ffn in ("none", "5+5", "10+10", "all26"):
        for att in ("none", "all26"):
            for lm in (False, True):
                name = f"ffn={ffn} att={att} lm={'int8' if lm else 'bf16'}"
                out[name] = make_mask(ffn, att, lm)
    return out


# Gemma-3-1B linear shapes [N, K] (output rows x input channels) and their bf16 sizes.
HIDDEN, INTER, VOCAB, N_Q, N_KV, HEAD_DIM = 1152, 6912, 262144, 4, 1, 256
LINEAR_SHAPES = {
    "qkv": ((N_Q + 2 * N_KV) * HEAD_DIM, HIDDEN),
    "o": (HIDDEN, N_Q * HEAD_DIM),
    "gate_up": (2 * INTER, HIDDEN),
    "down": (HIDDEN, INTER),
    "lm_head": (VOCAB, HIDDEN),
}


def weight_mib(name: str, bytes_per_elt: int = 2) -> float:
    n, k = LINEAR_SHAPES[name]
    return n * k * bytes_per_elt / 2**20
