"""Oracle for the fingerprint forward pass: plain, slow, CPU-only numpy code.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import it.  It shares no code with
the CUDA path (``paper_2501_13111_gb300``) and imports nothing from it; the
only module both sides use is ``synth`` (seeded input generation).

What it follows (arXiv 2501.13111, "iServe"):

* The fingerprint (Sec. 1; Sec. 5.1) is the LLM rebuilt with the same
  components -- embedding, hidden (decoder) layers, linear layers,
  normalisation, activation, softmax -- but only one or two hidden layers.
  The paper does not spell out the block; the reading used here is the
  Llama-2 decoder block (pre-norm RMSNorm, rotate-half RoPE, grouped-query
  attention, SwiGLU FFN, untied LM head, final RMSNorm).
* Deployment configurations (Sec. 2, Sec. 3.2; Table "Models and
  configurations"): INT8 and INT4 weight-only quantisation and an INT8 KV
  cache.  The paper names the formats only; the exact quantisers are the
  readings written out in ``quant.py``.
* The KV cache makes every decode step cost the same per token (Sec. 5.3,
  text before Eq. 1), and latency splits as Eq. 1-3; ``estimator.py``
  solves those systems.

Floating point: fp64 everywhere except where a quantiser's contract fixes
fp32 decisions (``quant.py``).  Parity of the full-model values is pinned
only through their pinned parts (tests/test_oracle_*.py): the paper prints
no worked example of a forward pass.
"""
from . import quant, model, memory, estimator  # noqa: F401
