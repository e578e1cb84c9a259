"""CPU oracle of the packed-cache attention step (test infrastructure only).

Imported by the tests, the smoke check and the benchmark's CPU baseline; never
by the library.  See kvq_oracle for what each function follows.
"""
from .kvq_oracle import *  # noqa: F401,F403
from .kvq_oracle import (OracleCache, affine_quant, symmetric_quant, pack_codes,  # noqa: F401
                         unpack_codes, fwht_f32, davn_f32, attention, attend,
                         project_lora, round_to, nf4_levels, nf4_dequant,
                         project_lora_nf4, attention_backward, lora_backward)
