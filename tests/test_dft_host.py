"""The register DFTs of the PAR kernels (csrc/dft.cuh, `__host__ __device__`) compiled for the
host with g++ and checked for every tile side 1..8 against numpy's FFT: the forward 2-D
real transform of an h x w tile (Section 4.3 applies RFFT2 per tile) and its inverse on a
Hermitian-consistent half spectrum.  No GPU is needed."""
import os
import shutil
import subprocess

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2609_34144_gb300", "csrc")

DRIVER = r"""
#define __host__
#define __device__
#define __forceinline__ inline
#include <cstdio>
#include "dft.cuh"
using namespace cast;
int main() {
  int h, w;
  while (std::scanf("%d %d", &h, &w) == 2) {
    float x[8][8] = {};
    for (int y = 0; y < h; ++y)
      for (int xx = 0; xx < w; ++xx) std::scanf("%f", &x[y][xx]);
    float re[8][5] = {}, im[8][5] = {};
    dft::fwd2d(x, h, w, re, im);
    for (int ky = 0; ky < h; ++ky)
      for (int kx = 0; kx <= w / 2; ++kx) std::printf("%.9g %.9g\n", re[ky][kx], im[ky][kx]);
    float z[8][8] = {};
    dft::inv2d(re, im, h, w, z);
    for (int y = 0; y < h; ++y)
      for (int xx = 0; xx < w; ++xx) std::printf("%.9g\n", z[y][xx]);
    // the row-emitting inverse of the blend kernels, on the same spectrum
    float r2[8][5] = {}, i2[8][5] = {}, e[8][8] = {};
    dft::fwd2d(x, h, w, r2, i2);
    dft::inv2d_emit(r2, i2, h, w, [&](int yy, const float* row) {
      for (int xx = 0; xx < w; ++xx) e[yy][xx] = row[xx];
    });
    for (int y = 0; y < h; ++y)
      for (int xx = 0; xx < w; ++xx) std::printf("%.9g\n", e[y][xx]);
  }
  return 0;
}
"""


@pytest.fixture(scope="module")
def driver(tmp_path_factory):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    d = tmp_path_factory.mktemp("dft")
    src = d / "drv.cpp"
    src.write_text(DRIVER)
    exe = d / "drv"
    subprocess.run([gxx, "-std=c++17", "-O1", "-I", CSRC, str(src), "-o", str(exe)], check=True,
                   capture_output=True, text=True)
    return str(exe)


SIDES = [(h, w) for h in range(1, 9) for w in range(1, 9)]


def test_register_dfts_match_numpy(driver):
    rng = np.random.default_rng(11)
    tiles = [rng.standard_normal((h, w)).astype(np.float32) for h, w in SIDES]
    inp = "".join(f"{h} {w}\n" + " ".join(f"{v:.9g}" for v in t.ravel()) + "\n"
                  for (h, w), t in zip(SIDES, tiles))
    out = subprocess.run([driver], input=inp, capture_output=True, text=True, check=True).stdout
    vals = np.array(out.split(), dtype=np.float64)
    pos = 0
    for (h, w), t in zip(SIDES, tiles):
        nb = h * (w // 2 + 1)
        spec = vals[pos:pos + 2 * nb].reshape(h, w // 2 + 1, 2)
        pos += 2 * nb
        ref = np.fft.rfft2(t.astype(np.float64))          # unnormalised, e^{-2 pi i k n / N}
        scale = np.sqrt(h * w) * np.max(np.abs(t))
        np.testing.assert_allclose(spec[..., 0], ref.real, atol=2e-6 * scale, err_msg=f"{h}x{w} re")
        np.testing.assert_allclose(spec[..., 1], ref.imag, atol=2e-6 * scale, err_msg=f"{h}x{w} im")
        for what in ("inv2d", "inv2d_emit"):
            back = vals[pos:pos + h * w].reshape(h, w)
            pos += h * w
            # unnormalised inverse: h * w times the input
            np.testing.assert_allclose(back, h * w * t, atol=4e-6 * h * w * np.max(np.abs(t)),
                                       err_msg=f"{h}x{w} {what}")
    assert pos == len(vals)
