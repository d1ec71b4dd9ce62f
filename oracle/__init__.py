"""Float64 CPU oracle for the RSLM residual codec and IVF-probe search.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path (the CUDA library and
its Python binding) imports, calls, links or executes anything in this
package.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline
legs of ``bench.py`` may use it.

The oracle is a plain, slow, step-by-step restatement of the method in the
paper "RSLM: Training-Free Vector Quantization for Approximate Nearest
Neighbor Search":

* ``constants``  -- static sign table S1/S2 and permutation P (Sec. 3.1.2),
  Gaussian Lloyd-Max codebooks (Sec. 3.2, Table "Rslm Codec Specifications"),
  the EVT constant E_max(D) (Sec. 3.2, eq. for s_initial) and the UE7M9 /
  UE4M12 scale formats (Sec. 3.3.1, Sec. 3.5.2).
* ``rotation``   -- the block-wise cascaded FWHT rotation, materialised as an
  explicit D x D float64 matrix (Sec. 3.1.1-3.1.3).
* ``codec``      -- residual encoding with EVT scaling, nearest-codeword
  assignment, local and global norm correction (Sec. 3.2-3.5).
* ``search``     -- IVF probe by <q, centroid>, brute-force scoring of every
  probed candidate with the score identities of Sec. 3.5.1/3.5.2, full sorts,
  and rescoring from higher-bit codes (Sec. 5.5.1, Sec. 2.1).

Every function works in float64 with no blocking, fusion or reordering
beyond what the paper's definitions state.  Library primitives (matrix
products, sorts, quadrature) serve as single steps.

Parity pins: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, textbook values, invariants or brute force, except the
exact values of the 2-D and 4-D k-means codebooks, which are not unique
(any rotation of an optimum is optimal): "parity unpinned" for their exact
values; their optimality conditions (centroid condition, MSE below the
product code) are pinned.
"""
