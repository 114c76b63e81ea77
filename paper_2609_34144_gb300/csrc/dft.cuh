// Small 1-D and 2-D DFTs of tile sides 1..8 held entirely in registers (one channel per
// thread).  Lengths 8 and 4 use written-out radix-2 transforms and complex length 6 two
// length-3 transforms; the other lengths (edge tiles) use the defining sum with compile-time
// twiddles, zero twiddles left out.  Unnormalised: the caller folds the
// orthonormal 1/sqrt(h w) factors (Section 4.3, App. A.2) into its coefficients.
//
// Register layout of a tile spectrum: re[ky][kx], im[ky][kx] with ky < 8, kx < 5 (the
// stored half spectrum of an 8-wide tile); bins with ky >= h or kx > w/2 are unused.
#pragma once

namespace cast {
namespace dft {

// cos(2 pi m / N) and sin(2 pi m / N) for N = 1..8, m = 0..N-1 (mathematical constants).
__host__ __device__ __forceinline__ constexpr float tw_cos(int N, int m) {
  return
      (N == 1 && m == 0) ? 1.000000000e+00f :
      (N == 2 && m == 0) ? 1.000000000e+00f :
      (N == 2 && m == 1) ? -1.000000000e+00f :
      (N == 3 && m == 0) ? 1.000000000e+00f :
      (N == 3 && m == 1) ? -5.000000000e-01f :
      (N == 3 && m == 2) ? -5.000000000e-01f :
      (N == 4 && m == 0) ? 1.000000000e+00f :
      (N == 4 && m == 1) ? 0.000000000e+00f :
      (N == 4 && m == 2) ? -1.000000000e+00f :
      (N == 4 && m == 3) ? 0.000000000e+00f :
      (N == 5 && m == 0) ? 1.000000000e+00f :
      (N == 5 && m == 1) ? 3.090169944e-01f :
      (N == 5 && m == 2) ? -8.090169944e-01f :
      (N == 5 && m == 3) ? -8.090169944e-01f :
      (N == 5 && m == 4) ? 3.090169944e-01f :
      (N == 6 && m == 0) ? 1.000000000e+00f :
      (N == 6 && m == 1) ? 5.000000000e-01f :
      (N == 6 && m == 2) ? -5.000000000e-01f :
      (N == 6 && m == 3) ? -1.000000000e+00f :
      (N == 6 && m == 4) ? -5.000000000e-01f :
      (N == 6 && m == 5) ? 5.000000000e-01f :
      (N == 7 && m == 0) ? 1.000000000e+00f :
      (N == 7 && m == 1) ? 6.234898019e-01f :
      (N == 7 && m == 2) ? -2.225209340e-01f :
      (N == 7 && m == 3) ? -9.009688679e-01f :
      (N == 7 && m == 4) ? -9.009688679e-01f :
      (N == 7 && m == 5) ? -2.225209340e-01f :
      (N == 7 && m == 6) ? 6.234898019e-01f :
      (N == 8 && m == 0) ? 1.000000000e+00f :
      (N == 8 && m == 1) ? 7.071067812e-01f :
      (N == 8 && m == 2) ? 0.000000000e+00f :
      (N == 8 && m == 3) ? -7.071067812e-01f :
      (N == 8 && m == 4) ? -1.000000000e+00f :
      (N == 8 && m == 5) ? -7.071067812e-01f :
      (N == 8 && m == 6) ? 0.000000000e+00f :
      (N == 8 && m == 7) ? 7.071067812e-01f :
      0.0f;
}
__host__ __device__ __forceinline__ constexpr float tw_sin(int N, int m) {
  return
      (N == 1 && m == 0) ? 0.000000000e+00f :
      (N == 2 && m == 0) ? 0.000000000e+00f :
      (N == 2 && m == 1) ? 0.000000000e+00f :
      (N == 3 && m == 0) ? 0.000000000e+00f :
      (N == 3 && m == 1) ? 8.660254038e-01f :
      (N == 3 && m == 2) ? -8.660254038e-01f :
      (N == 4 && m == 0) ? 0.000000000e+00f :
      (N == 4 && m == 1) ? 1.000000000e+00f :
      (N == 4 && m == 2) ? 0.000000000e+00f :
      (N == 4 && m == 3) ? -1.000000000e+00f :
      (N == 5 && m == 0) ? 0.000000000e+00f :
      (N == 5 && m == 1) ? 9.510565163e-01f :
      (N == 5 && m == 2) ? 5.877852523e-01f :
      (N == 5 && m == 3) ? -5.877852523e-01f :
      (N == 5 && m == 4) ? -9.510565163e-01f :
      (N == 6 && m == 0) ? 0.000000000e+00f :
      (N == 6 && m == 1) ? 8.660254038e-01f :
      (N == 6 && m == 2) ? 8.660254038e-01f :
      (N == 6 && m == 3) ? 0.000000000e+00f :
      (N == 6 && m == 4) ? -8.660254038e-01f :
      (N == 6 && m == 5) ? -8.660254038e-01f :
      (N == 7 && m == 0) ? 0.000000000e+00f :
      (N == 7 && m == 1) ? 7.818314825e-01f :
      (N == 7 && m == 2) ? 9.749279122e-01f :
      (N == 7 && m == 3) ? 4.338837391e-01f :
      (N == 7 && m == 4) ? -4.338837391e-01f :
      (N == 7 && m == 5) ? -9.749279122e-01f :
      (N == 7 && m == 6) ? -7.818314825e-01f :
      (N == 8 && m == 0) ? 0.000000000e+00f :
      (N == 8 && m == 1) ? 7.071067812e-01f :
      (N == 8 && m == 2) ? 1.000000000e+00f :
      (N == 8 && m == 3) ? 7.071067812e-01f :
      (N == 8 && m == 4) ? 0.000000000e+00f :
      (N == 8 && m == 5) ? -7.071067812e-01f :
      (N == 8 && m == 6) ? -1.000000000e+00f :
      (N == 8 && m == 7) ? -7.071067812e-01f :
      0.0f;
}

constexpr float kRsqrt2 = 7.071067812e-01f;

// -------------------------------------------------------------- real forward, length N
// re[k] + i im[k] = sum_n x[n] exp(-2 pi i k n / N), k = 0..N/2
template <int N>
__host__ __device__ __forceinline__ void rfwd(const float* x, float* re, float* im) {
#pragma unroll
  for (int k = 0; k <= N / 2; ++k) {
    float ar = 0.f, ai = 0.f;
#pragma unroll
    for (int n = 0; n < N; ++n) {
      const float c = tw_cos(N, (k * n) % N), s = tw_sin(N, (k * n) % N);
      // zero twiddles skipped at compile time (x * 0 is not foldable under IEEE rules)
      if (c != 0.f) ar += x[n] * c;
      if (s != 0.f) ai -= x[n] * s;
    }
    re[k] = ar;
    im[k] = ai;
  }
}

template <>
__host__ __device__ __forceinline__ void rfwd<4>(const float* x, float* re, float* im) {
  const float s02 = x[0] + x[2], s13 = x[1] + x[3];
  re[0] = s02 + s13;      im[0] = 0.f;
  re[1] = x[0] - x[2];    im[1] = x[3] - x[1];
  re[2] = s02 - s13;      im[2] = 0.f;
}

template <>
__host__ __device__ __forceinline__ void rfwd<8>(const float* x, float* re, float* im) {
  const float es0 = x[0] + x[4], ed0 = x[0] - x[4], es1 = x[2] + x[6], ed1 = x[2] - x[6];
  const float os0 = x[1] + x[5], od0 = x[1] - x[5], os1 = x[3] + x[7], od1 = x[3] - x[7];
  const float E0 = es0 + es1, E2 = es0 - es1, O0 = os0 + os1, O2 = os0 - os1;
  const float u = (od0 - od1) * kRsqrt2, v = (od0 + od1) * kRsqrt2;
  re[0] = E0 + O0;  im[0] = 0.f;
  re[1] = ed0 + u;  im[1] = -ed1 - v;
  re[2] = E2;       im[2] = -O2;
  re[3] = ed0 - u;  im[3] = ed1 - v;
  re[4] = E0 - O0;  im[4] = 0.f;
}

// -------------------------------------------------------------- real inverse, length N
// x[n] = sum over the Hermitian extension of re/im[0..N/2] of X[k] exp(+2 pi i k n / N);
// the imaginary parts of the k = 0 and (N even) k = N/2 entries are ignored.
template <int N>
__host__ __device__ __forceinline__ void rinv(const float* re, const float* im, float* x) {
#pragma unroll
  for (int n = 0; n < N; ++n) {
    float acc = re[0];
    if (N % 2 == 0) acc += (n % 2 ? -re[N / 2] : re[N / 2]);
#pragma unroll
    for (int k = 1; k <= (N - 1) / 2; ++k) {
      const float c = 2.f * tw_cos(N, (k * n) % N), s = 2.f * tw_sin(N, (k * n) % N);
      if (c != 0.f) acc += re[k] * c;
      if (s != 0.f) acc -= im[k] * s;
    }
    x[n] = acc;
  }
}

template <>
__host__ __device__ __forceinline__ void rinv<4>(const float* re, const float* im, float* x) {
  const float e = re[0] + re[2], o = re[0] - re[2];
  x[0] = e + 2.f * re[1];
  x[2] = e - 2.f * re[1];
  x[1] = o - 2.f * im[1];
  x[3] = o + 2.f * im[1];
}

template <>
__host__ __device__ __forceinline__ void rinv<8>(const float* re, const float* im, float* x) {
  // even/odd output split: z_k = A_k + i B_k, x[2m] + i x[2m+1] = IDFT4(z)[m]
  const float A0 = re[0] + re[4], B0 = re[0] - re[4];
  const float A1r = re[1] + re[3], A1i = im[1] - im[3];
  const float D1r = re[1] - re[3], D1i = im[1] + im[3];
  const float B1r = (D1r - D1i) * kRsqrt2, B1i = (D1r + D1i) * kRsqrt2;
  const float z0r = A0, z0i = B0;
  const float z1r = A1r - B1i, z1i = A1i + B1r;
  const float z2r = 2.f * re[2], z2i = -2.f * im[2];
  const float z3r = A1r + B1i, z3i = -A1i + B1r;
  const float t0r = z0r + z2r, t0i = z0i + z2i, t1r = z0r - z2r, t1i = z0i - z2i;
  const float t2r = z1r + z3r, t2i = z1i + z3i, t3r = z1r - z3r, t3i = z1i - z3i;
  x[0] = t0r + t2r;  x[1] = t0i + t2i;   // y0
  x[4] = t0r - t2r;  x[5] = t0i - t2i;   // y2
  x[2] = t1r - t3i;  x[3] = t1i + t3r;   // y1 = t1 + i t3
  x[6] = t1r + t3i;  x[7] = t1i - t3r;   // y3 = t1 - i t3
}

// -------------------------------------------------------------- complex, length N, column kx
// In place on column `kx` of [8][5] arrays: X[k] = sum_n x[n] exp(SIGN 2 pi i k n / N).
template <int N, int SIGN, int KX>
__host__ __device__ __forceinline__ void ccol(float (&re)[8][5], float (&im)[8][5]) {
  float xr[N], xi[N];
#pragma unroll
  for (int n = 0; n < N; ++n) { xr[n] = re[n][KX]; xi[n] = im[n][KX]; }
#pragma unroll
  for (int k = 0; k < N; ++k) {
    float ar = 0.f, ai = 0.f;
#pragma unroll
    for (int n = 0; n < N; ++n) {
      const float c = tw_cos(N, (k * n) % N), s = SIGN * tw_sin(N, (k * n) % N);
      if (c != 0.f) {
        ar += xr[n] * c;
        ai += xi[n] * c;
      }
      if (s != 0.f) {
        ar -= xi[n] * s;
        ai += xr[n] * s;
      }
    }
    re[k][KX] = ar;
    im[k][KX] = ai;
  }
}

template <int SIGN>
__host__ __device__ __forceinline__ void fft4(float& a0r, float& a0i, float& a1r, float& a1i,
                                              float& a2r, float& a2i, float& a3r, float& a3i) {
  const float t0r = a0r + a2r, t0i = a0i + a2i, t1r = a0r - a2r, t1i = a0i - a2i;
  const float t2r = a1r + a3r, t2i = a1i + a3i, t3r = a1r - a3r, t3i = a1i - a3i;
  // SIGN i t3 = (-SIGN t3i, SIGN t3r)
  a0r = t0r + t2r;  a0i = t0i + t2i;
  a2r = t0r - t2r;  a2i = t0i - t2i;
  a1r = t1r - SIGN * t3i;  a1i = t1i + SIGN * t3r;
  a3r = t1r + SIGN * t3i;  a3i = t1i - SIGN * t3r;
}

template <int SIGN, int KX>
__host__ __device__ __forceinline__ void ccol8(float (&re)[8][5], float (&im)[8][5]) {
  float er[4] = {re[0][KX], re[2][KX], re[4][KX], re[6][KX]};
  float ei[4] = {im[0][KX], im[2][KX], im[4][KX], im[6][KX]};
  float orr[4] = {re[1][KX], re[3][KX], re[5][KX], re[7][KX]};
  float oi[4] = {im[1][KX], im[3][KX], im[5][KX], im[7][KX]};
  fft4<SIGN>(er[0], ei[0], er[1], ei[1], er[2], ei[2], er[3], ei[3]);
  fft4<SIGN>(orr[0], oi[0], orr[1], oi[1], orr[2], oi[2], orr[3], oi[3]);
  // W^k O[k], W = exp(SIGN 2 pi i / 8) = (1 + SIGN i) / sqrt 2
  float wr[4], wi[4];
  wr[0] = orr[0];  wi[0] = oi[0];
  wr[1] = (orr[1] - SIGN * oi[1]) * kRsqrt2;  wi[1] = (oi[1] + SIGN * orr[1]) * kRsqrt2;
  wr[2] = -SIGN * oi[2];  wi[2] = SIGN * orr[2];
  wr[3] = (-orr[3] - SIGN * oi[3]) * kRsqrt2;  wi[3] = (-oi[3] + SIGN * orr[3]) * kRsqrt2;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    re[k][KX] = er[k] + wr[k];      im[k][KX] = ei[k] + wi[k];
    re[k + 4][KX] = er[k] - wr[k];  im[k + 4][KX] = ei[k] - wi[k];
  }
}

template <int SIGN, int KX>
__host__ __device__ __forceinline__ void ccol4(float (&re)[8][5], float (&im)[8][5]) {
  fft4<SIGN>(re[0][KX], im[0][KX], re[1][KX], im[1][KX], re[2][KX], im[2][KX], re[3][KX], im[3][KX]);
}

// Length 3: A0 = a + b + c, A1,2 = a - (b + c) / 2 +- SIGN i (sqrt 3 / 2)(b - c).
template <int SIGN>
__host__ __device__ __forceinline__ void dft3(float& ar, float& ai, float& br, float& bi, float& cr,
                                              float& ci) {
  constexpr float kHalfSqrt3 = 8.660254038e-01f;
  const float tr = br + cr, ti = bi + ci, ur = br - cr, ui = bi - ci;
  const float mr = ar - 0.5f * tr, mi = ai - 0.5f * ti;
  // SIGN i (sqrt 3 / 2) u
  const float vr = -SIGN * kHalfSqrt3 * ui, vi = SIGN * kHalfSqrt3 * ur;
  ar = ar + tr;  ai = ai + ti;
  br = mr + vr;  bi = mi + vi;
  cr = mr - vr;  ci = mi - vi;
}

// Length 6 by decimation in time: two length-3 transforms of the even and odd samples,
// X[k] = E[k] + w^k O[k], X[k + 3] = E[k] - w^k O[k], w = exp(SIGN 2 pi i / 6).
template <int SIGN, int KX>
__host__ __device__ __forceinline__ void ccol6(float (&re)[8][5], float (&im)[8][5]) {
  constexpr float kHalfSqrt3 = 8.660254038e-01f;
  float e0r = re[0][KX], e0i = im[0][KX], e1r = re[2][KX], e1i = im[2][KX], e2r = re[4][KX], e2i = im[4][KX];
  float o0r = re[1][KX], o0i = im[1][KX], o1r = re[3][KX], o1i = im[3][KX], o2r = re[5][KX], o2i = im[5][KX];
  dft3<SIGN>(e0r, e0i, e1r, e1i, e2r, e2i);
  dft3<SIGN>(o0r, o0i, o1r, o1i, o2r, o2i);
  // w = 1/2 + SIGN i sqrt3/2, w^2 = -1/2 + SIGN i sqrt3/2
  const float w1r = 0.5f * o1r - SIGN * kHalfSqrt3 * o1i, w1i = 0.5f * o1i + SIGN * kHalfSqrt3 * o1r;
  const float w2r = -0.5f * o2r - SIGN * kHalfSqrt3 * o2i, w2i = -0.5f * o2i + SIGN * kHalfSqrt3 * o2r;
  re[0][KX] = e0r + o0r;  im[0][KX] = e0i + o0i;
  re[3][KX] = e0r - o0r;  im[3][KX] = e0i - o0i;
  re[1][KX] = e1r + w1r;  im[1][KX] = e1i + w1i;
  re[4][KX] = e1r - w1r;  im[4][KX] = e1i - w1i;
  re[2][KX] = e2r + w2r;  im[2][KX] = e2i + w2i;
  re[5][KX] = e2r - w2r;  im[5][KX] = e2i - w2i;
}

template <int N, int SIGN, int KX>
__host__ __device__ __forceinline__ void col(float (&re)[8][5], float (&im)[8][5]) {
  if constexpr (N == 8) ccol8<SIGN, KX>(re, im);
  else if constexpr (N == 6) ccol6<SIGN, KX>(re, im);
  else if constexpr (N == 4) ccol4<SIGN, KX>(re, im);
  else ccol<N, SIGN, KX>(re, im);
}

// A column whose row transforms are real: kx = 0, and kx = w/2 for even w (the only width
// with a fifth stored column is w = 8, whose column 4 is its Nyquist column).  Forward
// (SIGN = -1) it holds a real signal: a real transform gives ky = 0..N/2 and the mirrors
// N - ky follow by conjugation.  Inverse (SIGN = +1) it holds the Hermitian spectrum of a
// real signal (the conjugate-symmetric blend of App. A.2): the real inverse reads
// ky = 0..N/2 only and the imaginary parts of the result are zero.
template <int N, int SIGN, int KX>
__host__ __device__ __forceinline__ void rcol(float (&re)[8][5], float (&im)[8][5]) {
  if constexpr (SIGN < 0) {
    float x[N], r[N / 2 + 1], i[N / 2 + 1];
#pragma unroll
    for (int n = 0; n < N; ++n) x[n] = re[n][KX];
    rfwd<N>(x, r, i);
#pragma unroll
    for (int k = 0; k <= N / 2; ++k) {
      re[k][KX] = r[k];
      im[k][KX] = i[k];
    }
#pragma unroll
    for (int k = 1; k <= (N - 1) / 2; ++k) {
      re[N - k][KX] = r[k];
      im[N - k][KX] = -i[k];
    }
  } else {
    float r[N / 2 + 1], i[N / 2 + 1], x[N];
#pragma unroll
    for (int k = 0; k <= N / 2; ++k) {
      r[k] = re[k][KX];
      i[k] = im[k][KX];
    }
    rinv<N>(r, i, x);
#pragma unroll
    for (int n = 0; n < N; ++n) {
      re[n][KX] = x[n];
      im[n][KX] = 0.f;
    }
  }
}

// -------------------------------------------------------------- 2-D, tile h x w
template <int W>
__host__ __device__ __forceinline__ void rows_fwd(const float (&x)[8][8], int h, float (&re)[8][5],
                                                  float (&im)[8][5]) {
#pragma unroll
  for (int y = 0; y < 8; ++y)
    if (y < h) rfwd<W>(x[y], re[y], im[y]);
}
template <int H, int SIGN>
__host__ __device__ __forceinline__ void cols(int w, float (&re)[8][5], float (&im)[8][5]) {
  const int nkx = w / 2;
  rcol<H, SIGN, 0>(re, im);
  if (nkx >= 1) col<H, SIGN, 1>(re, im);
  if (nkx >= 2) col<H, SIGN, 2>(re, im);
  if (nkx >= 3) col<H, SIGN, 3>(re, im);
  if (nkx >= 4) rcol<H, SIGN, 4>(re, im);
}
template <int W>
__host__ __device__ __forceinline__ void rows_inv(const float (&re)[8][5], const float (&im)[8][5],
                                                  int h, float (&x)[8][8]) {
#pragma unroll
  for (int y = 0; y < 8; ++y)
    if (y < h) rinv<W>(re[y], im[y], x[y]);
}

// Unnormalised forward 2-D real DFT of the h x w tile in x (1 <= h, w <= 8).
__host__ __device__ __forceinline__ void fwd2d(const float (&x)[8][8], int h, int w,
                                               float (&re)[8][5], float (&im)[8][5]) {
  switch (w) {
    case 8: rows_fwd<8>(x, h, re, im); break;
    case 7: rows_fwd<7>(x, h, re, im); break;
    case 6: rows_fwd<6>(x, h, re, im); break;
    case 5: rows_fwd<5>(x, h, re, im); break;
    case 4: rows_fwd<4>(x, h, re, im); break;
    case 3: rows_fwd<3>(x, h, re, im); break;
    case 2: rows_fwd<2>(x, h, re, im); break;
    default: rows_fwd<1>(x, h, re, im); break;
  }
  switch (h) {
    case 8: cols<8, -1>(w, re, im); break;
    case 7: cols<7, -1>(w, re, im); break;
    case 6: cols<6, -1>(w, re, im); break;
    case 5: cols<5, -1>(w, re, im); break;
    case 4: cols<4, -1>(w, re, im); break;
    case 3: cols<3, -1>(w, re, im); break;
    case 2: cols<2, -1>(w, re, im); break;
    default: cols<1, -1>(w, re, im); break;
  }
}

template <int W, class Emit>
__host__ __device__ __forceinline__ void rows_inv_emit(const float (&re)[8][5], const float (&im)[8][5],
                                                       int h, Emit&& emit) {
#pragma unroll
  for (int y = 0; y < 8; ++y) {
    if (y < h) {
      float row[8];
      rinv<W>(re[y], im[y], row);
      emit(y, row);
    }
  }
}

// Unnormalised inverse of fwd2d, handing each output row (W values) to emit(y, row) as soon
// as it is formed (destroys re/im).
template <class Emit>
__host__ __device__ __forceinline__ void inv2d_emit(float (&re)[8][5], float (&im)[8][5], int h,
                                                    int w, Emit&& emit) {
  switch (h) {
    case 8: cols<8, 1>(w, re, im); break;
    case 7: cols<7, 1>(w, re, im); break;
    case 6: cols<6, 1>(w, re, im); break;
    case 5: cols<5, 1>(w, re, im); break;
    case 4: cols<4, 1>(w, re, im); break;
    case 3: cols<3, 1>(w, re, im); break;
    case 2: cols<2, 1>(w, re, im); break;
    default: cols<1, 1>(w, re, im); break;
  }
  switch (w) {
    case 8: rows_inv_emit<8>(re, im, h, emit); break;
    case 7: rows_inv_emit<7>(re, im, h, emit); break;
    case 6: rows_inv_emit<6>(re, im, h, emit); break;
    case 5: rows_inv_emit<5>(re, im, h, emit); break;
    case 4: rows_inv_emit<4>(re, im, h, emit); break;
    case 3: rows_inv_emit<3>(re, im, h, emit); break;
    case 2: rows_inv_emit<2>(re, im, h, emit); break;
    default: rows_inv_emit<1>(re, im, h, emit); break;
  }
}

// Unnormalised inverse of fwd2d for a Hermitian-consistent half spectrum (destroys re/im).
__host__ __device__ __forceinline__ void inv2d(float (&re)[8][5], float (&im)[8][5], int h, int w,
                                               float (&x)[8][8]) {
  switch (h) {
    case 8: cols<8, 1>(w, re, im); break;
    case 7: cols<7, 1>(w, re, im); break;
    case 6: cols<6, 1>(w, re, im); break;
    case 5: cols<5, 1>(w, re, im); break;
    case 4: cols<4, 1>(w, re, im); break;
    case 3: cols<3, 1>(w, re, im); break;
    case 2: cols<2, 1>(w, re, im); break;
    default: cols<1, 1>(w, re, im); break;
  }
  switch (w) {
    case 8: rows_inv<8>(re, im, h, x); break;
    case 7: rows_inv<7>(re, im, h, x); break;
    case 6: rows_inv<6>(re, im, h, x); break;
    case 5: rows_inv<5>(re, im, h, x); break;
    case 4: rows_inv<4>(re, im, h, x); break;
    case 3: rows_inv<3>(re, im, h, x); break;
    case 2: rows_inv<2>(re, im, h, x); break;
    default: rows_inv<1>(re, im, h, x); break;
  }
}

}  // namespace dft
}  // namespace cast
