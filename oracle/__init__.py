"""fp64 CPU oracle for the Ms. Forcing MSSA/MSP window pass.

TEST INFRASTRUCTURE ONLY. Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import anything here. The product path
(the CUDA library and its Python binding) never calls into this package and
shares no code with it.

Everything is plain numpy in float64, written from the paper:
  schedule.py  Eq. 3 token counts, Eq. 4 context enumeration, Eq. 5 ratio
  mssa.py      Eq. 4 context construction (explicit resampled K/V) and naive
               softmax attention
  msp.py       MSP patchify / unpatchify with optional tier projections
  stream.py    rolling-window history update (Sec. 3.1, Algorithm 1)
  brute.py     a second, per-query enumeration of Eq. 4 for tiny grids
  mssa_bwd.py  the gradient of Eq. 4 (softmax Jacobian and the adjoint of
               Subsample), for training through the window

Readings of points the paper leaves open (all chosen once, used everywhere):
  * Subsample: AVG (s x s block mean, the default) or STRIDED (top-left pick).
  * V(a) holds every history frame and every window position, a included.
  * History frames are fine-scale; the sink is never resampled.
  * Context order: sink, history frames in slot order, window states 1..T.
  * Softmax scale 1/sqrt(D), no mask, no positional encoding.
  * Patch feature order (c, dy, dx); tokens row-major over the state grid.
"""
