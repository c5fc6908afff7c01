"""The oracle's thread-parallel row driver returns exactly what the serial one does."""
import numpy as np

from oracle import oracle as O
from synthetic import workloads as w
from synthetic.workloads import Shape


def test_parallel_rows_equal_serial_rows(oracle_lib):
    shape = Shape("par", 2, 6, 2, 64, 96, 1.0e4)
    hist, chunk = 40, 24
    q, k, v = w.tokens(shape, "par", chunk)
    kc, vc = w.cache(shape, "par", hist, fill="random")
    O.append(shape, k, v, hist, kc, vc, lib=oracle_lib)
    rows = np.array([(b, i, h) for b in range(shape.batch) for i in range(chunk) for h in range(shape.n_q_heads)],
                    np.int32)
    serial = O.attend_rows(shape, q, hist, kc, vc, rows, lib=oracle_lib)
    for threads in (1, 3, 7):
        par = O.attend_rows_parallel(shape, q, hist, kc, vc, rows, threads=threads, lib=oracle_lib)
        assert (par == serial).all()
