"""Float64 CPU oracle for the FLARE++ routing chain -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import this package. It shares no code with the CUDA library and never calls it; the
CUDA library never calls it either.

What it computes (FLARE++ paper):
  * ``sdpa``           -- SDPA(Q, K, V) = softmax(s Q K^T) V over the keys (Sec. 2, eq. sdpa_definition)
  * ``route``          -- Q = SDPA(Qseed, Kt, Vt); Z = SDPA(Q, K, V); Y = SDPA(K, Q, Z)
                          (Sec. 3.2, eqs. flarepp_dynamic_query and flarepp_mixer)
  * ``flare``          -- Z = SDPA(Q_h, K, V); Y = SDPA(K, Q_h, Z) with learned queries Q_h
                          shared by the batch (Sec. 3, eq. prelim_flare_sdpa)
  * ``encode_sharded`` -- the encoder evaluated shard by shard, then merged by the stable
                          log-sum-exp reduction (App. A.2, A.3)
  * ``mixer``          -- the FLARE++ token-mixing layer (Fig. 1; eqs. flarepp_query_synthesis
                          and flarepp_mixer): K, V, K~, V~ = X W^T split into heads, the routing
                          chain, then O = merge(Y) Wo^T; the projections are numpy matmuls
  * ``mixer_bwd``      -- the mixer layer's gradients: dO through the output projection (a
                          numpy matmul), the chain's backward (``route_bwd``), the projections'
                          weight gradients and dX (numpy matmuls)
  * ``sdpa_bwd``       -- the backward of one SDPA from its saved output and log-normaliser
                          (App. A.5): P = exp(S - L), c = <dO, O>, dV = P^T dO,
                          dS = P o (dO V^T - c), dK = s dS^T Q, dQ = s dS K
  * ``route_bwd``      -- the chain's backward: calls 3, 2, 1 in turn, the decoder's query
                          gradient added to call 2's before call 1, the seeds' gradient
                          summed over the batch (App. A.5)

All arithmetic is float64 in ``flarepp_oracle.c``; this module only marshals numpy arrays.
"""
import ctypes

import numpy as np

from . import build as _build

_c_i64 = ctypes.c_int64
_c_dp = ctypes.POINTER(ctypes.c_double)


class Oracle:
    """One loaded build of the oracle library (``plant`` != 0 only in pin-strength tests)."""

    def __init__(self, plant: int = 0, build_dir: str = _build.BUILD_DIR):
        path = _build.build(plant, build_dir)
        self.lib = ctypes.CDLL(path)
        self.plant = plant
        lib = self.lib
        lib.oracle_sdpa_f64.restype = ctypes.c_int
        lib.oracle_sdpa_f64.argtypes = [_c_i64, _c_i64, _c_i64, _c_i64, _c_dp, ctypes.c_int,
                                        _c_dp, _c_dp, ctypes.c_double, _c_dp, _c_dp]
        lib.oracle_route_f64.restype = ctypes.c_int
        lib.oracle_route_f64.argtypes = [_c_i64] * 5 + [_c_dp] * 5 + [ctypes.c_double] + [_c_dp] * 3
        lib.oracle_encode_sharded_f64.restype = ctypes.c_int
        lib.oracle_encode_sharded_f64.argtypes = [_c_i64] * 4 + [_c_dp] * 3 + [
            ctypes.c_double, _c_i64, _c_i64, _c_dp, _c_dp]
        lib.oracle_sdpa_bwd_f64.restype = ctypes.c_int
        lib.oracle_sdpa_bwd_f64.argtypes = [_c_i64] * 4 + [_c_dp] * 6 + [ctypes.c_double] + [
            _c_dp] * 3
        lib.oracle_route_bwd_f64.restype = ctypes.c_int
        lib.oracle_route_bwd_f64.argtypes = [_c_i64] * 5 + [_c_dp] * 5 + [ctypes.c_double] + [
            _c_dp] * 6
        lib.oracle_max_threads.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        assert lib.oracle_plant() == plant

    # ------------------------------------------------------------------ helpers
    @staticmethod
    def _f64(a):
        return np.ascontiguousarray(np.asarray(a, dtype=np.float64))

    @staticmethod
    def _p(a):
        return a.ctypes.data_as(_c_dp)

    def max_threads(self) -> int:
        return int(self.lib.oracle_max_threads())

    def set_threads(self, n: int) -> None:
        self.lib.oracle_set_threads(int(n))

    # ------------------------------------------------------------------ API
    def sdpa(self, q, k, v, scale):
        """SDPA over the last two axes. q [..., nq, D]; k, v [..., nk, D] (same leading shape).

        Returns (out [..., nq, D], lse [..., nq]); a row with no keys gives out 0, lse -inf.
        """
        q, k, v = self._f64(q), self._f64(k), self._f64(v)
        lead = q.shape[:-2]
        assert k.shape[:-2] == lead and v.shape == k.shape and q.shape[-1] == k.shape[-1]
        G = int(np.prod(lead)) if lead else 1
        nq, D = q.shape[-2], q.shape[-1]
        nk = k.shape[-2]
        out = np.zeros(lead + (nq, D))
        lse = np.zeros(lead + (nq,))
        rc = self.lib.oracle_sdpa_f64(G, nq, nk, D, self._p(q), 0, self._p(k), self._p(v),
                                      float(scale), self._p(out), self._p(lse))
        if rc:
            raise MemoryError("oracle scratch allocation failed")
        return out, lse

    def route(self, seeds, Kt, Vt, K, V, scale):
        """The routing chain. seeds [H, M, D]; Kt, Vt, K, V [B, H, N, D].

        Returns (Q [B, H, M, D], Z [B, H, M, D], Y [B, H, N, D]).
        """
        seeds, Kt, Vt, K, V = (self._f64(a) for a in (seeds, Kt, Vt, K, V))
        B, H, N, D = K.shape
        M = seeds.shape[1]
        assert seeds.shape == (H, M, D)
        for a in (Kt, Vt, V):
            assert a.shape == (B, H, N, D)
        Q = np.zeros((B, H, M, D))
        Z = np.zeros((B, H, M, D))
        Y = np.zeros((B, H, N, D))
        rc = self.lib.oracle_route_f64(B, H, N, M, D, self._p(seeds), self._p(Kt), self._p(Vt),
                                       self._p(K), self._p(V), float(scale), self._p(Q),
                                       self._p(Z), self._p(Y))
        if rc:
            raise MemoryError("oracle scratch allocation failed")
        return Q, Z, Y

    def flare(self, Q, K, V, scale):
        """FLARE with learned queries (Sec. 3, eq. prelim_flare_sdpa): per (b, h), the encoder
        Z = SDPA(Q_h, K, V) and the decoder Y = SDPA(K, Q_h, Z), both this oracle's SDPA.
        Q [H, M, D] is shared by the batch; K, V [B, H, N, D].

        Returns (Z [B, H, M, D], Y [B, H, N, D]).
        """
        Q, K, V = self._f64(Q), self._f64(K), self._f64(V)
        B, H, N, D = K.shape
        assert Q.shape[0] == H and Q.shape[2] == D and V.shape == K.shape
        Qb = np.ascontiguousarray(np.broadcast_to(Q, (B,) + Q.shape))
        Z, _ = self.sdpa(Qb, K, V, scale)
        Y, _ = self.sdpa(K, Qb, Z, scale)
        return Z, Y

    def mixer(self, X, W_in, Wo, seeds, scale):
        """The FLARE++ mixer (Fig. 1): X [B, N, C]; W_in [P*C, C] in the out x in layout, its
        row blocks the projections of K, V, K~, V~ (P = 4; P = 2 ties K~, V~ to K, V, the
        shared-projection variant of App. C.2); Wo [C, C] (out x in); seeds [H, M, D] with
        C = H * D. Returns O [B, N, C]."""
        X, W_in, Wo, seeds = (self._f64(a) for a in (X, W_in, Wo, seeds))
        B, N, C = X.shape
        H, M, D = seeds.shape
        assert H * D == C and W_in.shape[1] == C and W_in.shape[0] in (2 * C, 4 * C)
        assert Wo.shape == (C, C)
        proj = X @ W_in.T  # [B, N, P*C]: the pointwise projections of eq. flarepp_mixer

        def heads(i):  # block i of the projection, split into H heads of width D
            blk = proj[..., i * C:(i + 1) * C].reshape(B, N, H, D)
            return np.ascontiguousarray(blk.transpose(0, 2, 1, 3))

        K, V = heads(0), heads(1)
        Kt, Vt = (heads(2), heads(3)) if W_in.shape[0] == 4 * C else (K, V)
        _, _, Y = self.route(seeds, Kt, Vt, K, V, scale)
        merged = Y.transpose(0, 2, 1, 3).reshape(B, N, C)  # merge(Y): heads side by side
        return merged @ Wo.T

    def mixer_bwd(self, X, W_in, Wo, seeds, scale, dO):
        """Gradients of ``mixer`` for the output gradient dO [B, N, C]: returns
        (dX [B, N, C], dW_in [P*C, C], dWo [C, C], dseeds [H, M, D]). With P = 2 the projections
        of K~, V~ are those of K, V, so each block collects both gradients."""
        X, W_in, Wo, seeds, dO = (self._f64(a) for a in (X, W_in, Wo, seeds, dO))
        B, N, C = X.shape
        H, M, D = seeds.shape
        P = W_in.shape[0] // C
        proj = X @ W_in.T

        def heads(T):  # [B, N, C] -> [B, H, N, D]
            return np.ascontiguousarray(T.reshape(B, N, H, D).transpose(0, 2, 1, 3))

        def merge(T):  # [B, H, N, D] -> [B, N, C]
            return T.transpose(0, 2, 1, 3).reshape(B, N, C)

        K, V = heads(proj[..., :C]), heads(proj[..., C:2 * C])
        Kt, Vt = (heads(proj[..., 2 * C:3 * C]), heads(proj[..., 3 * C:])) if P == 4 else (K, V)
        _, _, Y = self.route(seeds, Kt, Vt, K, V, scale)
        Ym = merge(Y)
        # O = merge(Y) Wo^T
        dWo = np.einsum("bno,bni->oi", dO, Ym)
        dY = heads(dO @ Wo)
        dseeds, dKt, dVt, dK, dV = self.route_bwd(seeds, Kt, Vt, K, V, scale, dY)
        blocks = [dK, dV, dKt, dVt] if P == 4 else [dK + dKt, dV + dVt]
        dproj = np.concatenate([merge(g) for g in blocks], axis=-1)  # [B, N, P*C]
        # proj = X W_in^T
        dW_in = np.einsum("bnr,bnc->rc", dproj, X)
        dX = dproj @ W_in
        return dX, dW_in, dWo, dseeds

    def sdpa_bwd(self, q, k, v, out, lse, dout, scale):
        """Backward of ``sdpa`` (App. A.5) from the forward's ``out`` and ``lse``.

        q, out, dout [..., nq, D]; k, v [..., nk, D]; lse [..., nq].
        Returns (dq, dk, dv) shaped like q, k, v.
        """
        q, k, v, out, lse, dout = (self._f64(a) for a in (q, k, v, out, lse, dout))
        lead = q.shape[:-2]
        assert k.shape[:-2] == lead and v.shape == k.shape and out.shape == q.shape
        assert dout.shape == q.shape and lse.shape == q.shape[:-1]
        G = int(np.prod(lead)) if lead else 1
        nq, D = q.shape[-2], q.shape[-1]
        nk = k.shape[-2]
        dq, dk, dv = np.zeros(q.shape), np.zeros(k.shape), np.zeros(v.shape)
        rc = self.lib.oracle_sdpa_bwd_f64(G, nq, nk, D, self._p(q), self._p(k), self._p(v),
                                          self._p(out), self._p(lse), self._p(dout),
                                          float(scale), self._p(dq), self._p(dk), self._p(dv))
        if rc:
            raise MemoryError("oracle scratch allocation failed")
        return dq, dk, dv

    def route_bwd(self, seeds, Kt, Vt, K, V, scale, dY):
        """Gradients of the routing chain for the output gradient dY [B, H, N, D].

        Returns (dseeds [H, M, D], dKt, dVt, dK, dV [B, H, N, D]).
        """
        seeds, Kt, Vt, K, V, dY = (self._f64(a) for a in (seeds, Kt, Vt, K, V, dY))
        B, H, N, D = K.shape
        M = seeds.shape[1]
        assert seeds.shape == (H, M, D)
        for a in (Kt, Vt, V, dY):
            assert a.shape == (B, H, N, D)
        dseeds = np.zeros((H, M, D))
        grads = [np.zeros((B, H, N, D)) for _ in range(4)]
        rc = self.lib.oracle_route_bwd_f64(B, H, N, M, D, self._p(seeds), self._p(Kt),
                                           self._p(Vt), self._p(K), self._p(V), float(scale),
                                           self._p(dY), self._p(dseeds),
                                           *(self._p(g) for g in grads))
        if rc:
            raise MemoryError("oracle scratch allocation failed")
        return (dseeds, *grads)

    def encode_sharded(self, q, k, v, scale, chunk, n_empty=0):
        """Encoder over shards of ``chunk`` keys merged by the stable LSE reduction (App. A.3).

        q [..., nq, D]; k, v [..., nk, D]. ``n_empty`` extra empty shards are merged in.
        Returns (out [..., nq, D], lse [..., nq]).
        """
        q, k, v = self._f64(q), self._f64(k), self._f64(v)
        lead = q.shape[:-2]
        G = int(np.prod(lead)) if lead else 1
        nq, D = q.shape[-2], q.shape[-1]
        nk = k.shape[-2]
        out = np.zeros(lead + (nq, D))
        lse = np.zeros(lead + (nq,))
        rc = self.lib.oracle_encode_sharded_f64(G, nq, nk, D, self._p(q), self._p(k), self._p(v),
                                                float(scale), int(chunk), int(n_empty),
                                                self._p(out), self._p(lse))
        if rc:
            raise ValueError("oracle_encode_sharded_f64 failed (chunk <= 0 or allocation)")
        return out, lse


_default = None


def default() -> Oracle:
    global _default
    if _default is None:
        _default = Oracle(0)
    return _default


def sdpa(q, k, v, scale):
    return default().sdpa(q, k, v, scale)


def route(seeds, Kt, Vt, K, V, scale):
    return default().route(seeds, Kt, Vt, K, V, scale)


def flare(Q, K, V, scale):
    return default().flare(Q, K, V, scale)


def encode_sharded(q, k, v, scale, chunk, n_empty=0):
    return default().encode_sharded(q, k, v, scale, chunk, n_empty)


def mixer(X, W_in, Wo, seeds, scale):
    return default().mixer(X, W_in, Wo, seeds, scale)


def mixer_bwd(X, W_in, Wo, seeds, scale, dO):
    return default().mixer_bwd(X, W_in, Wo, seeds, scale, dO)


def sdpa_bwd(q, k, v, out, lse, dout, scale):
    return default().sdpa_bwd(q, k, v, out, lse, dout, scale)


def route_bwd(seeds, Kt, Vt, K, V, scale, dY):
    return default().route_bwd(seeds, Kt, Vt, K, V, scale, dY)


def max_threads() -> int:
    return default().max_threads()


def set_threads(n: int) -> None:
    default().set_threads(n)


def build() -> str:
    """Compile the oracle library (called by the package build step)."""
    return _build.build()


__all__ = ["Oracle", "default", "sdpa", "route", "flare", "encode_sharded", "mixer",
           "mixer_bwd", "sdpa_bwd", "route_bwd", "max_threads", "set_threads", "build"]
