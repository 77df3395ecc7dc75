"""CPU oracle for CacheReforge bounded KV-cache recomputation.

TEST INFRASTRUCTURE ONLY. This package is the plain, slow, obviously-correct
restatement of what the recomputation path computes. Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference arm may
import it; the product library never does, and it shares no code with the CUDA
path (the two meet only in the seeded input generator, ``synth``).

Layout:

* ``decoder``  -- one Qwen2.5-style decoder layer under base weights plus an
  unmerged LoRA adapter (Eq. S1, Eq. S3; the block itself is the standard
  pre-norm decoder of the model family named in Section 5.1).
* ``cache``    -- the versioned, paged, layerwise KV cache (Eq. 1), fresh
  prefill, executable window restart (Section 4.2) and the first-step
  next-token logits of a hybrid cache (Section 3.1, Section S1.2).
* ``fidelity`` -- forward KL at the first generated-token step (Section S2.1),
  top-1 agreement, tail influence and its certificates (Eq. 2, 4, 5; derived in
  Section S1.2).
* ``drift``    -- adapter displacement per layer and module (Eq. 8), dense and
  rank-factored.
* ``policy``   -- host recovery policy: invalidation onset (Eq. S4), candidate
  windows, labels (Eq. 6), sensitivity (Eq. 7), runtime risk (Eq. 8), range end
  (Eq. 9), anchor update (Section 4.2).

Precision: layer arithmetic runs in the dtype passed as ``dt`` (float32 by
default, float64 in the pins); norms' mean-square, softmax normalisation, KL and
drift accumulate in float64. Parameters arrive as the bf16 values the GPU gets,
upcast, so input quantisation is not counted as error.

Parity pins (tests/test_oracle_*.py): merged == unmerged LoRA and the alpha / r
scale; brute-force and library attention; library RMSNorm/SiLU; complex-number
RoPE; a whole decoder layer against a composition of torch library ops with
merged weights; the final norm + LM head and the embedding lookup against
torch; window(0, N) == prefill; identical adapters reproduce the stale cache; a
one-layer window after a query/output/MLP update leaves that layer's K/V
unchanged (Eq. S4); tail decode over a fresh cache gives the fresh logits; KL
identities and the Eq. 4 / Eq. 5 certificates; factored == dense drift; policy
worked examples printed in the paper (tests/golden/). Every function here has
at least one such pin. The paper prints no worked example of K/V/H values for
its models, so those values are pinned through the library composition at
small sizes and through identities that hold at any size, not through stored
numbers.
"""
from . import decoder, cache, fidelity, drift, policy  # noqa: F401
