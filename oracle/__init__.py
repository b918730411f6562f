"""CPU fp64 oracle of Dynamic Memory Compression (Nawrot et al., ICML 2024).

TEST INFRASTRUCTURE ONLY. Nothing on the product path may import, link or run
anything in this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it. It shares no
code with the CUDA path (``paper_2403_09636_gb300``) and imports nothing from it.

Modules:
  dmc_ref   -- numpy fp64 definitions: gates (Eq. reuse), the single-head cache
               update (Algorithm 1), decode attention (Eq. attn-softmax over the
               compressed cache), the closed form of a prompt's slots (segment
               means of Eq. partial-accumulation with binary alpha) and the
               training-time masked formulation (Eq. partial-accumulation plus the
               additive mask of the masking figure and the masking appendix);
               prompt-phase attention (each prompt token over the closed slots
               and its own running state); the window-grouping approximation of
               Sec. 3.3 (window = w) in the update, the closed form and the
               masked formulation.
  cref      -- ctypes loader for dmc_ref.c, the same Algorithm 1 plus attention in
               plain C (fp64), used for timed CPU baselines and for parity at sizes
               where numpy's per-token loop is too slow.
"""
