"""The worker-sharded context semantics of include/asap.h restated on the
oracle (fp64), so that the exchange plan and the per-round protocol of
paper_1612_08608_gb300.sharded can be checked on the CPU with gloo ranks.
Test infrastructure only."""
import numpy as np

from oracle import rounds, sgd


class OracleShardContext:
    row_dtype = np.float64

    def __init__(self, shards, B, loss, lr, k, graph_kind, graph_seed=0, regenerate=False):
        self.sh, self.B, self.loss, self.lr, self.k = shards, B, loss, lr, k
        self.N, self.P = shards.N, shards.d
        self.sched = rounds.graph_schedule(graph_kind, self.N, k, graph_seed, regenerate)
        self.W = np.zeros((self.N, self.P))
        self.t = 0
        self.first, self.count = 0, self.N
        self.pending = False
        self.delivered = set()

    def set_worker_range(self, first, count):
        self.first, self.count = first, count

    def own(self, j):
        return self.first <= j < self.first + self.count

    def get_graph(self, rnd):
        nbr, wgt = self.sched(rnd)
        return np.asarray(nbr, np.int32), np.asarray(wgt, np.float64)

    def local_step(self):
        assert not self.pending
        for i in range(self.first, self.first + self.count):
            self.W[i], _, _ = sgd.sparse_worker_step(self.W[i], self.sh.rowptr[i], self.sh.col[i], self.sh.val[i],
                                                     self.sh.y[i], self.t, self.B, self.loss, self.lr)
        self.delivered = set()
        self.pending = True

    def read_rows(self, rows):
        return self.W[np.asarray(rows)].copy(), 1.0

    def write_rows(self, rows, values):
        assert self.pending
        for j, v in zip(rows, values):
            assert not self.own(int(j))
            self.W[int(j)] = v
            self.delivered.add(int(j))

    def stochastic_reduce(self):
        nbr, wgt = self.get_graph(self.t)
        own = range(self.first, self.first + self.count)
        for i in own:
            for j in nbr[i]:
                if not self.own(int(j)) and int(j) not in self.delivered:
                    raise RuntimeError("in-neighbour %d of worker %d not delivered" % (j, i))
        out = self.W.copy()
        for i in own:
            out[i] = sum(float(wgt[i, m]) * self.W[int(nbr[i, m])] for m in range(nbr.shape[1]))
        self.W = out
        self.t += 1
        self.pending = False
