"""The five synthetic workloads the kernels are measured and tested on.

Shapes come from the paper's models: GPT-2 small (Section 3.1, Exp. 5:
12 heads, r = 192/12 = 16, d_v = 64), Mistral-7B (Section 3.5, Exp. 8:
32 query / 8 kv heads, rank 256 = 32 per kv head, d_v = 128) and a 7B MHA
model trained with d_select = d_model/4 (Section 3.2, Exp. 7: 32 heads,
r = 32, d_v = 128).  All tensors are N(0, 1) rounded to bf16 and the scale
is 1/sqrt(r).
"""

from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class Workload:
    name: str
    kind: str            # "decode", "prefill" or "layer"
    batch: int
    h_q: int
    h_kv: int
    r: int
    d_v: int
    seq: int = 0          # context (decode) or prompt length (prefill)
    seq_range: tuple = ()  # ragged contexts: uniform integers in [lo, hi]
    page_size: int = 0
    k_int8: bool = False
    decode_steps: int = 0
    seed: int = 1000
    notes: str = ""
    r_sweep: tuple = field(default_factory=tuple)
    cached: int = 0       # prefill of a chunk after this many cached tokens

    def as_config(self) -> dict:
        d = {"workload": self.name, "batch": self.batch, "h_q": self.h_q, "h_kv": self.h_kv,
             "r": self.r, "d_v": self.d_v}
        if self.seq:
            d["seq"] = self.seq
        if self.seq_range:
            d["seq_range"] = list(self.seq_range)
        if self.page_size:
            d["page_size"] = self.page_size
        if self.cached:
            d["cached"] = self.cached
        d["k_dtype"] = "int8" if self.k_int8 else "bf16"
        return d


GPT2_LAYER = Workload("gpt2_small_layer_prefill256_decode32", "layer", 1, 12, 12, 16, 64, seq=256,
                      decode_steps=32, seed=1000,
                      notes="causal prefill S=256 then 32 decode steps appending to a contiguous cache, fp32 out")
MISTRAL_GQA_DECODE = Workload("mistral7b_gqa_decode_b16_ctx4096", "decode", 16, 32, 8, 32, 128,
                              seq=4096, seed=1001)
MHA7B_PREFILL = Workload("mha7b_causal_prefill_b2_s8192", "prefill", 2, 32, 32, 32, 128, seq=8192,
                         seed=1002, notes="bf16 output")
# Chunked prefill (a serving engine's prompt chunk): 4096 new tokens of the 7B
# shape after 4096 cached ones, the keys read back from a contiguous cache.
CHUNKED_PREFILL = Workload("mha7b_chunked_prefill_b2_4096_after_4096", "prefill", 2, 32, 32, 32, 128,
                           seq=4096, cached=4096, seed=1006, notes="bf16 output")
PAGED_LONG_DECODE = Workload("paged_decode_b4_ctx64k_128k", "decode", 4, 32, 8, 32, 128,
                             seq_range=(65536, 131072), page_size=64, seed=1003)
INT8_DECODE = Workload("int8_key_decode_b64_ctx32768", "decode", 64, 32, 8, 32, 128, seq=32768,
                       k_int8=True, seed=1004, r_sweep=(16, 32, 64, 128))

ALL = (GPT2_LAYER, MISTRAL_GQA_DECODE, MHA7B_PREFILL, PAGED_LONG_DECODE, INT8_DECODE)
