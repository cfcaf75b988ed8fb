"""Plain fp64 CPU oracle of SPIDER's accelerated prefill, written from the paper.

TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may
import this package. The CUDA path never imports it, and it never imports the CUDA path.

* prune.py: MSV-Prune (§4.1, Eq. 1-3).
* decoder.py: decoder prefill with VSkip-Attn / VSkip-FFN bypass (§3.2, §4.2-4.3, Alg. 1).
"""
