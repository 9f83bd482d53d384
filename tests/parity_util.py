"""Helpers for the GPU parity tests: run a layer through the C ABI and the
CPU oracle on the same seeded inputs and compare.

Tolerances (stated per output, spec contract):
  codes   bit-exact
  alpha   |a_gpu - a_orc| <= 1e-6 |a_orc|
  conv / linear, fp32 output, no epilogue:
          |y_gpu - y_orc| <= 2e-3 * bound,  bound = |alpha| * sum|x| over the
          receptive field (the oracle returns it with y)
  bf16 output adds the output rounding: + 2^-8 |y_orc| (one bf16 ulp is at
          most 2^-7 |y| relative; half of it is the rounding error, doubled
          for margin); an epilogue (residual, ReLU) adds 2^-22 |y_orc|.
"""
import numpy as np
import torch

import oracle
import paper_1701_00485_gb300 as tbn

TOL_BOUND = 2e-3
ALPHA_RTOL = 1e-6


def u32(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().numpy().view(np.uint32)


def check_quantize(W2d_cpu: torch.Tensor, codes_gpu, alpha_gpu, rows=None):
    """Compare GPU codes/alpha with the oracle for the given rows (all if None)."""
    W = W2d_cpu.numpy()
    if rows is not None:
        W = W[rows]
        codes = u32(codes_gpu)[rows]
        alpha = alpha_gpu.detach().cpu().numpy()[rows]
    else:
        codes = u32(codes_gpu)
        alpha = alpha_gpu.detach().cpu().numpy()
    wt, al = oracle.quantize(W)
    want = oracle.pack(wt)
    bad = np.argwhere(codes != want)
    assert bad.size == 0, "codes differ at %s (gpu %08x, oracle %08x)" % (
        bad[0].tolist(), int(codes[tuple(bad[0])]), int(want[tuple(bad[0])]))
    err = np.abs(alpha.astype(np.float64) - al)
    lim = ALPHA_RTOL * np.abs(al)
    assert np.all(err <= lim), "alpha rel err %.3g at row %d" % (
        float(np.max(err / np.maximum(np.abs(al), 1e-300))), int(np.argmax(err - lim)))


def assert_within(y_gpu: np.ndarray, y_orc: np.ndarray, bound: np.ndarray, out_bf16: bool,
                  epilogue: bool = False, what: str = "", extra: float = 0.0):
    """|gpu - oracle| <= (TOL_BOUND + extra) * bound, plus the bf16 rounding of
    the output when out_bf16 (extra: a further relative error per term the
    path is allowed, e.g. 2^-9 for an operand rounded to bf16)."""
    y_gpu = y_gpu.astype(np.float64)
    tol = (TOL_BOUND + extra) * bound
    if out_bf16:
        tol = tol + 2.0 ** -8 * np.abs(y_orc)
    if epilogue:
        tol = tol + 2.0 ** -22 * np.abs(y_orc)
    err = np.abs(y_gpu - y_orc)
    ok = err <= tol
    if not np.all(ok):
        i = np.unravel_index(np.argmax(err - tol), err.shape)
        raise AssertionError("%s: %d/%d outside tolerance; worst at %s gpu=%r oracle=%r bound=%r"
                             % (what, int((~ok).sum()), ok.size, tuple(int(v) for v in i),
                                float(y_gpu[i]), float(y_orc[i]), float(bound[i])))
    return float(np.max(err / np.maximum(bound, 1e-300)))


class ConvCase:
    """One conv layer: fp32 weights [K,C,R,S], activations NCHW (cpu)."""

    def __init__(self, x_nchw: torch.Tensor, W: torch.Tensor, stride, pad):
        self.x = x_nchw
        self.W = W
        self.stride = tuple(stride)
        self.pad = tuple(pad)
        self.K, self.C, self.R, self.S = W.shape

    def quantize_gpu(self, layout):
        # codes in (r, s, c) order for NHWC and NCHW_NHWC, (c, r, s) for NCHW
        if layout != tbn.TBN_NCHW:
            Wl = self.W.permute(0, 2, 3, 1).reshape(self.K, -1).contiguous()
        else:
            Wl = self.W.reshape(self.K, -1).contiguous()
        codes, alpha = tbn.tbn_quantize_pack(Wl.cuda())
        return Wl, codes, alpha

    def run_gpu(self, layout, x_dtype, out_dtype, algo=tbn.TBN_CONV_AUTO, relu=False,
                residual=None):
        Wl, codes, alpha = self.quantize_gpu(layout)
        check_quantize(Wl, codes, alpha)
        x = self.x.to(x_dtype)
        if layout == tbn.TBN_NHWC:
            x = x.permute(0, 2, 3, 1).contiguous()
        res = None
        y_nhwc = layout != tbn.TBN_NCHW
        if residual is not None:
            res = residual.to(out_dtype)
            if y_nhwc:
                res = res.permute(0, 2, 3, 1).contiguous()
            res = res.cuda()
        y = tbn.tbn_conv2d_fwd(x.cuda(), codes, alpha, self.K, self.R, self.S, self.stride,
                               self.pad, layout=layout, out_dtype=out_dtype, relu=relu,
                               residual=res, algo=algo)
        torch.cuda.synchronize()
        y = y.float().cpu()
        if y_nhwc:
            y = y.permute(0, 3, 1, 2).contiguous()
        return y.numpy()

    def oracle_full(self, x_dtype):
        x = self.x.to(x_dtype).float().numpy()
        wt, al = oracle.quantize(self.W.reshape(self.K, -1).numpy())
        return oracle.conv2d_nchw(x, wt.reshape(self.K, self.C, self.R, self.S), al,
                                  self.stride, self.pad)

    def oracle_sites(self, x_dtype, sites):
        x = self.x.to(x_dtype).float().numpy()
        wt, al = oracle.quantize(self.W.reshape(self.K, -1).numpy())
        return oracle.conv2d_sites(x, wt.reshape(self.K, self.C, self.R, self.S), al, sites,
                                   self.stride, self.pad)


def random_sites(shape, count, seed):
    rng = np.random.default_rng(seed)
    cols = [rng.integers(0, d, size=count) for d in shape]
    # always include the corners of the output (ragged tiles, padding)
    corners = []
    for b in (0, shape[0] - 1):
        for k in (0, shape[1] - 1):
            for p in (0, shape[2] - 1):
                for q in (0, shape[3] - 1):
                    corners.append((b, k, p, q))
    s = np.stack(cols, axis=1)
    return np.concatenate([np.array(corners, dtype=np.int64), s.astype(np.int64)], axis=0)
