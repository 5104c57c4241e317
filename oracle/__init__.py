"""CPU oracle for the hybrid packed-CKKS linear layer (Fiona, Sec. 4.2).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers.  The product path
(``paper_2609_35352_gb300``) never imports, links or runs anything here.

Contents
  oracle.c       schoolbook modular evaluation of the layer (flat and DAG form,
                 and with plaintext scale classes)
  rescale.c      negacyclic NTT (by definition and radix-2) and the rescale by
                 the last prime that follows the layer
  encode.c       plaintext encoding: slots -> integer coefficients by the
                 inversion formula of the canonical embedding, and integer
                 coefficients -> RNS NTT form
  crt.py         brute-force evaluation over Z_Q with Python integers (pin P2)
  ckks_tiny.py   tiny-N CKKS encode/encrypt/decrypt round trip (pin P3)

Pins (tests/test_oracle_pins.py): every function here is checked against
something other than itself -- the worked example of Sec. 4.2, exact
distributivity (hybrid == all-PMult with t*gamma plaintexts), CRT over the
full modulus Q, a CKKS round trip against a float64 slot-wise mat-vec,
special cases with closed forms, and a planted-mistake check.
"""
from .liboracle import build, linear_eval, linear_eval_classes, linear_eval_dag, load, load_variant  # noqa: F401
from .liboracle import intt, min_root, ntt, rescale  # noqa: F401
from .liboracle import ckks_embed, encode_coeffs  # noqa: F401
