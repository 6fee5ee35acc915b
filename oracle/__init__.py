"""CPU oracle for the SDSAT block decode step -- TEST INFRASTRUCTURE ONLY.

A plain, slow, obviously correct reference of what the CUDA path computes.
Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline/reference
arm may import it; the product package never does, and it shares no code
with the CUDA path (the only common dependency is `synth`, which produces
inputs and holds none of the method's arithmetic).

Contents
--------
model     Llama-architecture decoder block forward of q new positions against
          a KV cache (the P_theta(. | context) of the paper's Eq. 1-2), fp64.
sampling  argmax with the lowest-id tie break, the fixed-point nucleus
          (top-p) sampler, the exp used by it, and Philox4x32-10.
decode    Eq. 3 verification, the two-step-draft-then-verify loops (greedy,
          and chain-form nucleus, Sec. 2.1.2) and plain decoding loops.
tree      the tree-structured draft step 2 (Sec. 2.1.2): tree forward with
          depth positions and ancestor masks, longest accepted branch, KV
          compaction, the tree decoding loop.
pipelined the pipelined variant (not a step of the paper): the verification
          block also carries the adaptive tokens, so a loop whose drafts are
          all accepted needs no separate draft step 1.

Pins (tests/test_oracle_*.py) tie every function to something other than
itself: closed forms, invariants the method fixes (greedy SDSAT output equals
plain greedy output, Sec. 2.1.1; a q-row block equals q sequential steps),
brute force on tiny inputs and published known-answer vectors; the decoder
forward's composition is pinned on weight settings where it reduces to library
routines (zeroed branches, a single key, one causal attention layer).  The
end-to-end logits of a randomly initialised model with every branch on have no
printed values anywhere: beyond those pins they are "parity unpinned".
"""
