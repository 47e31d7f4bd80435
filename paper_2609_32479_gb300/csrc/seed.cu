// Analytic seed of Sec. 3.1 on the GPU, in fp64: per track the helix through
// three hits (conformal map), its perigee, and per hit the three residual
// features against that helix (asinh du, asinh dv in the curvilinear frame,
// path length s); plus the decode of the heads' corrections against the seed
// (Sec. 3.3).  One thread per track: the work per track is a few hundred fp64
// operations and transcendental calls, and tracks are independent.
//
// Conventions (those of the synthetic track generator): B along +z; a positive
// charge turns clockwise seen from +z; at turning angle a from the perigee the
// direction angle is phi0 - q a, the transverse arc length R a and
// z = z0 + R a cot(theta); the perigee point is (-d0 sin phi0, d0 cos phi0);
// p_T = 0.299792458 B R / 1000 GeV (R in mm, B in T); q/p = q sin(theta) / p_T.
#include <math.h>

#include "trackfit_internal.h"

namespace {

constexpr double C_LIGHT = 0.299792458;
constexpr double TWO_PI = 6.283185307179586476925286766559;
constexpr double PI = 3.1415926535897932384626433832795;
constexpr double QOP_FLOOR = 0.02;   // 1/GeV: floor of the scale-free q/p residual (Sec. 3.3)
constexpr int NEWTON_MAX = 60;
constexpr double PITCH_MIN_MM = 1.0;   // below this pitch z does not choose the helix turn of a hit

// x mod 2 pi in [0, 2 pi)
__device__ __forceinline__ double mod2pi(double x) {
  double r = fmod(x, TWO_PI);
  return r < 0.0 ? r + TWO_PI : r;
}

struct Helix {
  double d0, z0, phi0, theta, qop;
  double q, R, cx, cy, x0, y0, g0, st, ct;
};

// Geometry of the helix of a perigee (centre, radius, angle of the perigee point
// around the centre).
__device__ Helix helix_of(const double (&pg)[5], double b_field) {
  Helix h;
  h.d0 = pg[0];
  h.z0 = pg[1];
  h.phi0 = pg[2];
  h.theta = pg[3];
  h.qop = pg[4];
  h.q = h.qop > 0.0 ? 1.0 : (h.qop < 0.0 ? -1.0 : 0.0);
  h.st = sin(h.theta);
  h.ct = cos(h.theta);
  h.R = 1000.0 * h.st / fabs(h.qop) / (C_LIGHT * b_field);
  double sp, cp;
  sincos(h.phi0, &sp, &cp);
  h.x0 = -h.d0 * sp;
  h.y0 = h.d0 * cp;
  h.cx = h.x0 + h.q * h.R * sp;
  h.cy = h.y0 - h.q * h.R * cp;
  h.g0 = atan2(h.y0 - h.cy, h.x0 - h.cx);
  return h;
}

// Perigee of the helix through three hits in path order (Sec. 3.1: the circle
// from the conformal map, whose image of a circle through the first hit is a
// straight line fixed by the images of the other two).
__device__ void perigee_from_triplet(const double (&a)[3], const double (&b)[3], const double (&c)[3],
                                     double b_field, double (&pg)[5]) {
  const double ax = b[0] - a[0], ay = b[1] - a[1];
  const double bx = c[0] - a[0], by = c[1] - a[1];
  const double na = ax * ax + ay * ay, nb = bx * bx + by * by;
  const double u1 = ax / na, v1 = ay / na, u2 = bx / nb, v2 = by / nb;
  const double det = u1 * v2 - u2 * v1;
  const double ccx = (v2 - v1) / (2.0 * det), ccy = (u1 - u2) / (2.0 * det);
  const double Cx = a[0] + ccx, Cy = a[1] + ccy;
  const double R = hypot(ccx, ccy);
  const double cross = ax * by - ay * bx;
  const double q = cross > 0.0 ? -1.0 : (cross < 0.0 ? 1.0 : 0.0);
  const double dc = hypot(Cx, Cy);
  const double ux = Cx / dc, uy = Cy / dc;
  const double px = Cx - R * ux, py = Cy - R * uy;     // circle point closest to the beam line
  const double tx = -q * uy, ty = q * ux;              // direction of motion there
  const double phi0 = atan2(ty, tx);
  double sp, cp;
  sincos(phi0, &sp, &cp);
  const double d0 = -px * sp + py * cp;
  const double g_p = atan2(py - Cy, px - Cx);
  const double s0 = R * mod2pi(-q * (atan2(a[1] - Cy, a[0] - Cx) - g_p));
  const double s2 = R * mod2pi(-q * (atan2(c[1] - Cy, c[0] - Cx) - g_p));
  const double cot = (c[2] - a[2]) / (s2 - s0);
  const double z0 = a[2] - s0 * cot;
  const double theta = atan2(1.0, cot);
  const double pt = C_LIGHT * b_field * R / 1000.0;
  pg[0] = d0;
  pg[1] = z0;
  pg[2] = phi0;
  pg[3] = theta;
  pg[4] = q * sin(theta) / pt;
}

// (du, dv, s) of a hit against the helix: the foot point is the helix point whose
// normal plane holds the hit, found by Newton's method on g(a) = (hit - p(a)) . t(a).
// The start is the hit's transverse angle around the centre counted from the
// perigee into [-pi, pi) (continuous across the perigee), moved by the whole
// turns that bring it closest to the angle of the hit's z, (z - z0) / (R cot theta),
// where the pitch 2 pi R |cot theta| exceeds PITCH_MIN_MM.  du, dv are the hit's
// coordinates along U = z x t / |z x t| and V = t x U at the foot point,
// s = R a / sin(theta) (negative behind the perigee).
__device__ void residuals(const Helix& h, const double (&x)[3], double& du, double& dv, double& s) {
  const double cot = h.ct / h.st;
  double a = mod2pi(-h.q * (atan2(x[1] - h.cy, x[0] - h.cx) - h.g0) + PI) - PI;
  const double rcot = h.R / tan(h.theta);
  if (2.0 * PI * fabs(rcot) > PITCH_MIN_MM) a += TWO_PI * floor(((x[2] - h.z0) / rcot - a) / TWO_PI + 0.5);
  double px = 0.0, py = 0.0, pz = 0.0, tx = 0.0, ty = 0.0, tz = h.ct, sphi = 0.0, cphi = 1.0;
  auto at = [&](double aa) {
    sincos(h.phi0 - h.q * aa, &sphi, &cphi);
    px = h.cx - h.q * h.R * sphi;
    py = h.cy + h.q * h.R * cphi;
    pz = h.z0 + h.R * aa * cot;
    tx = h.st * cphi;
    ty = h.st * sphi;
  };
  for (int it = 0; it < NEWTON_MAX; ++it) {
    at(a);
    const double rx = x[0] - px, ry = x[1] - py, rz = x[2] - pz;
    const double g = rx * tx + ry * ty + rz * tz;
    // dp/da = (R / sin theta) t;  dt/da = q sin(theta) (sin phi, -cos phi, 0)
    const double dg = -h.R / h.st + (rx * h.q * h.st * sphi - ry * h.q * h.st * cphi);
    const double an = a - g / dg;
    const bool done = fabs(an - a) <= 1e-15 * fmax(1.0, fabs(a));
    a = an;
    if (done) break;
  }
  at(a);
  // U = z x t / |z x t| = (-t_y, t_x, 0) / sin(theta); V = t x U
  const double ux = -ty / h.st, uy = tx / h.st;
  const double vx = -tz * uy, vy = tz * ux, vz = tx * uy - ty * ux;
  const double rx = x[0] - px, ry = x[1] - py, rz = x[2] - pz;
  du = rx * ux + ry * uy;
  dv = rx * vx + ry * vy + rz * vz;
  s = h.R * a / h.st;
}

__global__ void seed_kernel(const float* __restrict__ hits, int hs, const int32_t* __restrict__ n_hits, int64_t B,
                            int T, double b_field, double min_sep, double* __restrict__ seed, float* __restrict__ feats,
                            int fs) {
  const int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (b >= B) return;
  int n = n_hits[b];
  if (n < 0) n = 0;
  if (n > T) n = 0;   // not a track: no seed
  const float* hb = hits + (size_t)b * T * hs;   // hit t of this track at hb[t * hs]
  // the seed triplet: the first hit, then each first later hit more than min_sep
  // (3-D) from the previous seed hit
  int pick[3] = {-1, -1, -1};
  int np = 0;
  double last[3] = {0.0, 0.0, 0.0};
  for (int t = 0; t < n && np < 3; ++t) {
    const double p[3] = {(double)hb[t * hs + 0], (double)hb[t * hs + 1], (double)hb[t * hs + 2]};
    bool take = np == 0;
    if (!take) {
      const double dx = p[0] - last[0], dy = p[1] - last[1], dz = p[2] - last[2];
      take = sqrt(dx * dx + dy * dy + dz * dz) > min_sep;
    }
    if (take) {
      pick[np++] = t;
      last[0] = p[0];
      last[1] = p[1];
      last[2] = p[2];
    }
  }
  double pg[5];
  const bool ok = np == 3;
  if (ok) {
    double h3[3][3];
    for (int k = 0; k < 3; ++k)
      for (int c = 0; c < 3; ++c) h3[k][c] = (double)hb[pick[k] * hs + c];
    perigee_from_triplet(h3[0], h3[1], h3[2], b_field, pg);
  } else {
    for (int k = 0; k < 5; ++k) pg[k] = __longlong_as_double(0x7ff8000000000000ll);
  }
  for (int k = 0; k < 5; ++k) seed[b * 5 + k] = pg[k];
  if (!feats) return;
  float* fo = feats + (size_t)b * T * fs;
  bool finite = ok;
  for (int k = 0; k < 5; ++k) finite = finite && isfinite(pg[k]);
  const Helix h = finite ? helix_of(pg, b_field) : Helix{};
  for (int t = 0; t < T; ++t) {
    float f0 = 0.0f, f1 = 0.0f, f2 = 0.0f;
    if (finite && t < n) {
      const double x[3] = {(double)hb[t * hs + 0], (double)hb[t * hs + 1], (double)hb[t * hs + 2]};
      double du, dv, s;
      residuals(h, x, du, dv, s);
      f0 = (float)asinh(du);
      f1 = (float)asinh(dv);
      f2 = (float)s;
    }
    fo[t * fs + 0] = f0;
    fo[t * fs + 1] = f1;
    fo[t * fs + 2] = f2;
  }
}

// out = seed + correction, phi wrapped to (-pi, pi]; q/p from the scale-free
// residual: q/p = q/p_seed + r (|q/p_seed| + 0.02 / GeV)  (Sec. 3.3).
__global__ void decode_kernel(const double* __restrict__ seed, const float* __restrict__ corr, int64_t B,
                              float* __restrict__ out) {
  const int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (b >= B) return;
  double v[5];
  for (int k = 0; k < 5; ++k) v[k] = seed[b * 5 + k] + (double)corr[b * 5 + k];
  v[2] = PI - mod2pi(PI - v[2]);
  v[4] = seed[b * 5 + 4] + (double)corr[b * 5 + 4] * (fabs(seed[b * 5 + 4]) + QOP_FLOOR);
  for (int k = 0; k < 5; ++k) out[b * 5 + k] = (float)v[k];
}

}  // namespace

extern "C" int trackfit_seed(const float* hits, int32_t hit_stride, const int32_t* n_hits, int64_t n_tracks,
                             int32_t max_hits, double b_field, double* seed_out, float* features_out,
                             int32_t feat_stride, void* stream) {
  tf_nvtx_range nvtx_range("trackfit_seed");
  if (!hits || !n_hits || !seed_out || n_tracks <= 0 || max_hits < 1 || max_hits > TF_MAX_HITS) {
    return TRACKFIT_ERR_INVALID_ARG;
  }
  if (hit_stride < 3 || (features_out && feat_stride < 3)) return TRACKFIT_ERR_INVALID_ARG;
  if (!(b_field > 0.0) || !isfinite(b_field)) return TRACKFIT_ERR_INVALID_ARG;
  const uintptr_t mis = reinterpret_cast<uintptr_t>(hits) | reinterpret_cast<uintptr_t>(seed_out) |
                        reinterpret_cast<uintptr_t>(n_hits) | reinterpret_cast<uintptr_t>(features_out);
  if (mis & 15u) return TRACKFIT_ERR_INVALID_ARG;
  const unsigned grid = (unsigned)((n_tracks + 127) / 128);
  seed_kernel<<<grid, 128, 0, reinterpret_cast<cudaStream_t>(stream)>>>(hits, hit_stride, n_hits, n_tracks, max_hits,
                                                                        b_field, 10.0, seed_out, features_out,
                                                                        feat_stride);
  return cudaPeekAtLastError() == cudaSuccess ? TRACKFIT_OK : TRACKFIT_ERR_CUDA;
}

extern "C" int trackfit_decode(const double* seed, const float* corrections, int64_t n_tracks, float* out_params,
                               void* stream) {
  tf_nvtx_range nvtx_range("trackfit_decode");
  if (!seed || !corrections || !out_params || n_tracks <= 0) return TRACKFIT_ERR_INVALID_ARG;
  const uintptr_t mis = reinterpret_cast<uintptr_t>(seed) | reinterpret_cast<uintptr_t>(corrections) |
                        reinterpret_cast<uintptr_t>(out_params);
  if (mis & 15u) return TRACKFIT_ERR_INVALID_ARG;
  const unsigned grid = (unsigned)((n_tracks + 255) / 256);
  decode_kernel<<<grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(seed, corrections, n_tracks, out_params);
  return cudaPeekAtLastError() == cudaSuccess ? TRACKFIT_OK : TRACKFIT_ERR_CUDA;
}
