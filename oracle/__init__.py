"""CPU oracle for SD^2 (steered speculative decoding) — TEST INFRASTRUCTURE ONLY.

A plain, slow, fp32 restatement of what the paper's method computes, used to check the
CUDA library. Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline arm may
import it; the product path (the C-ABI library and its Python binding) never does, and
shares no code with it: the only common module is the seeded input generator
(paper_2511_09844_gb300.workloads), which holds no step of the method's arithmetic.

Contents, each function citing the passage it restates:
  philox    Philox4x32-10 counter-based generator (Salmon et al., SC'11).
  fpmath    exp and log as fixed sequences of correctly rounded fp32 operations.
  sampling  softmax with an exact normaliser, exponential-race sampling, greedy and
            stochastic speculative acceptance (Sec. 3.1 "Verification"; Leviathan et al.).
  model     Llama-style pre-norm decoder forward with the steered SwiGLU of Eq. 2.
  steering  steering vector g_t = LN(W_hml [h_t, m_t, l_t]) and biases W_s g_t
            (Sec. 3.1, Eq. 2, App. A.2).
  sd        the draft-and-verify loop with KV bookkeeping (Sec. 3, Sec. 4 "Decoding").

Which functions are pinned by what is listed in each module's header.
"""
