// CPU oracle for the ABCD active-block step -- TEST INFRASTRUCTURE ONLY (see abcd_oracle.h).
//
// Plain fp64 code, one Gaussian / one pixel at a time, written from the definitions:
//   * Section 2 of the paper: block coordinate descent over spatial partitions; frozen
//     partitions in front of / behind the active one collapse into F and B by associativity
//     of "over"; each step renders the active block only, composites it with F and B,
//     evaluates the reconstruction loss and backpropagates into the active block only.
//   * 3D Gaussian Splatting (the renderer the paper instantiates, Section 1): EWA
//     projection J W Sigma W^T J^T + 0.3 I, 3-sigma tile rectangles on 16x16 tiles,
//     (tile, depth) ordering, alpha = min(0.99, o exp(-sigma)), skip alpha < 1/255,
//     stop before T would fall below 1e-4, real SH colour + 0.5 clamped at 0.
// Compiled with -ffp-contract=off so every double / float operation rounds once.
#include "abcd_oracle.h"

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

namespace {

constexpr double kPi = 3.14159265358979323846;

// ---------------------------------------------------------------------------------------
// Forward-mode dual numbers: value + derivative w.r.t. up to NT seeded inputs.
constexpr int NT = 59;   // 3 mean + 3 log-scale + 4 quat + 1 opacity logit + 16*3 SH

struct Dual {
  double v;
  double d[NT];
  Dual() : v(0.0) { std::memset(d, 0, sizeof d); }
  Dual(double x) : v(x) { std::memset(d, 0, sizeof d); }  // NOLINT (implicit on purpose)
};
inline Dual operator+(const Dual& a, const Dual& b) {
  Dual r; r.v = a.v + b.v; for (int i = 0; i < NT; ++i) r.d[i] = a.d[i] + b.d[i]; return r;
}
inline Dual operator-(const Dual& a, const Dual& b) {
  Dual r; r.v = a.v - b.v; for (int i = 0; i < NT; ++i) r.d[i] = a.d[i] - b.d[i]; return r;
}
inline Dual operator-(const Dual& a) {
  Dual r; r.v = -a.v; for (int i = 0; i < NT; ++i) r.d[i] = -a.d[i]; return r;
}
inline Dual operator*(const Dual& a, const Dual& b) {
  Dual r; r.v = a.v * b.v;
  for (int i = 0; i < NT; ++i) r.d[i] = a.d[i] * b.v + a.v * b.d[i];
  return r;
}
inline Dual operator/(const Dual& a, const Dual& b) {
  Dual r; r.v = a.v / b.v;
  const double ib = 1.0 / b.v;
  for (int i = 0; i < NT; ++i) r.d[i] = (a.d[i] - r.v * b.d[i]) * ib;
  return r;
}
inline Dual exp(const Dual& a) {
  Dual r; r.v = std::exp(a.v); for (int i = 0; i < NT; ++i) r.d[i] = r.v * a.d[i]; return r;
}
inline Dual sqrt(const Dual& a) {
  Dual r; r.v = std::sqrt(a.v);
  const double k = 0.5 / r.v;
  for (int i = 0; i < NT; ++i) r.d[i] = k * a.d[i];
  return r;
}
inline double val(const Dual& a) { return a.v; }
inline double val(double a) { return a; }
using std::exp;
using std::sqrt;

template <class S> S clamp_const(const S& x, double lo, double hi) {
  if (val(x) < lo) return S(lo);
  if (val(x) > hi) return S(hi);
  return x;
}

// ---------------------------------------------------------------------------------------
// Real spherical harmonics from their definition:
//   Y_l^0  = K_l^0 P_l(z)
//   Y_l^m  = sqrt2 K_l^m P_l^m(cos th) cos(m phi),   Y_l^-m = ... sin(m phi)   (m > 0)
//   K_l^m  = sqrt((2l+1)/(4 pi) (l-m)!/(l+m)!),
//   P_l^m(z) = (-1)^m (1-z^2)^(m/2) d^m P_l/dz^m   (Condon-Shortley phase),
// and (1-z^2)^(m/2) (cos m phi + i sin m phi) = (x + i y)^m on the unit sphere.
double factorial(int n) { double r = 1.0; for (int i = 2; i <= n; ++i) r *= i; return r; }

void legendre_coeffs(int l, double* c) {  // P_l(z) = sum_k c[k] z^k (Bonnet recursion)
  double p0[8] = {1.0}, p1[8] = {0.0, 1.0}, p2[8];
  if (l == 0) { std::memset(c, 0, 8 * sizeof(double)); c[0] = 1.0; return; }
  for (int k = 2; k < 8; ++k) p0[k] = 0.0;
  for (int k = 2; k < 8; ++k) p1[k] = 0.0;
  for (int n = 1; n < l; ++n) {   // (n+1) P_{n+1} = (2n+1) z P_n - n P_{n-1}
    for (int k = 0; k < 8; ++k) {
      const double zpn = (k > 0) ? p1[k - 1] : 0.0;
      p2[k] = ((2.0 * n + 1.0) * zpn - n * p0[k]) / (n + 1.0);
    }
    std::memcpy(p0, p1, sizeof p0);
    std::memcpy(p1, p2, sizeof p1);
  }
  std::memcpy(c, p1, 8 * sizeof(double));
}

template <class S> S sh_basis(int l, int m, const S& x, const S& y, const S& z) {
  const int am = m < 0 ? -m : m;
  double c[8];
  legendre_coeffs(l, c);
  S dp(0.0);                                  // d^am P_l / dz^am by Horner
  for (int k = l - am; k >= 0; --k)
    dp = dp * z + S(c[k + am] * factorial(k + am) / factorial(k));
  const double K = std::sqrt((2.0 * l + 1.0) / (4.0 * kPi) * factorial(l - am) / factorial(l + am));
  if (m == 0) return S(K) * dp;
  S re(1.0), im(0.0);
  for (int i = 0; i < am; ++i) {
    S nre = re * x - im * y;
    S nim = re * y + im * x;
    re = nre; im = nim;
  }
  const double cs = (am % 2) ? -1.0 : 1.0;
  const double k = std::sqrt(2.0) * K * cs;
  return (m > 0) ? S(k) * dp * re : S(k) * dp * im;
}

// ---------------------------------------------------------------------------------------
// Projection of one Gaussian (3DGS EWA splatting) in scalar type S.
template <class S> struct Proj {
  S u, v, ca, cb, cc, o, col[3], raw[3];
  double tz = 0, lam_max = 0, lam_min = 0, r_exact = 0, tan_x = 0, tan_y = 0;
  bool front = false;
};

template <class S>
void project_one(const S mu[3], const S ls[3], const S q[4], const S& logit, const S* sh,
                 int deg, const orc_camera& cam, const orc_opts& op, Proj<S>& P) {
  const double* R = cam.R;
  // camera-space mean t = R mu + t_cam
  S tx = S(R[0]) * mu[0] + S(R[1]) * mu[1] + S(R[2]) * mu[2] + S(cam.t[0]);
  S ty = S(R[3]) * mu[0] + S(R[4]) * mu[1] + S(R[5]) * mu[2] + S(cam.t[1]);
  S tz = S(R[6]) * mu[0] + S(R[7]) * mu[1] + S(R[8]) * mu[2] + S(cam.t[2]);
  P.tz = val(tz);
  P.front = val(tz) > op.near_z;
  if (!P.front) return;
  // world covariance Sigma = R(q) S S^T R(q)^T
  S s[3] = {exp(ls[0]), exp(ls[1]), exp(ls[2])};
  S qn = sqrt(q[0] * q[0] + q[1] * q[1] + q[2] * q[2] + q[3] * q[3]);
  S w = q[0] / qn, x = q[1] / qn, y = q[2] / qn, z = q[3] / qn;
  S Rq[3][3] = {
      {S(1.0) - S(2.0) * (y * y + z * z), S(2.0) * (x * y - w * z), S(2.0) * (x * z + w * y)},
      {S(2.0) * (x * y + w * z), S(1.0) - S(2.0) * (x * x + z * z), S(2.0) * (y * z - w * x)},
      {S(2.0) * (x * z - w * y), S(2.0) * (y * z + w * x), S(1.0) - S(2.0) * (x * x + y * y)}};
  S M[3][3];
  for (int i = 0; i < 3; ++i)
    for (int j = 0; j < 3; ++j) M[i][j] = Rq[i][j] * s[j];
  S Sig[3][3];
  for (int i = 0; i < 3; ++i)
    for (int j = 0; j < 3; ++j) {
      S acc(0.0);
      for (int k = 0; k < 3; ++k) acc = acc + M[i][k] * M[j][k];
      Sig[i][j] = acc;
    }
  // affine approximation of the perspective map at the mean (guarded x/z, y/z)
  const double limx = op.guard * (0.5 * cam.width / cam.fx);
  const double limy = op.guard * (0.5 * cam.height / cam.fy);
  S rx = tx / tz, ry = ty / tz;
  P.tan_x = val(rx);
  P.tan_y = val(ry);
  S xg = clamp_const(rx, -limx, limx) * tz;
  S yg = clamp_const(ry, -limy, limy) * tz;
  S J00 = S(cam.fx) / tz, J02 = S(-cam.fx) * xg / (tz * tz);
  S J11 = S(cam.fy) / tz, J12 = S(-cam.fy) * yg / (tz * tz);
  S T[2][3];
  for (int k = 0; k < 3; ++k) {
    T[0][k] = J00 * S(R[0 + k]) + J02 * S(R[6 + k]);
    T[1][k] = J11 * S(R[3 + k]) + J12 * S(R[6 + k]);
  }
  S C2[2][2];
  for (int i = 0; i < 2; ++i)
    for (int j = 0; j < 2; ++j) {
      S acc(0.0);
      for (int a = 0; a < 3; ++a)
        for (int b = 0; b < 3; ++b) acc = acc + T[i][a] * Sig[a][b] * T[j][b];
      C2[i][j] = acc;
    }
  S a = C2[0][0] + S(op.dilation), b = C2[0][1], c = C2[1][1] + S(op.dilation);
  S det = a * c - b * b;
  P.ca = c / det;
  P.cb = -b / det;
  P.cc = a / det;
  const double mid = 0.5 * (val(a) + val(c));
  const double disc = mid * mid - val(det);
  P.lam_max = mid + std::sqrt(std::max(0.1, disc));
  P.lam_min = mid - std::sqrt(std::max(0.0, disc));
  P.r_exact = 3.0 * std::sqrt(P.lam_max);
  P.u = S(cam.fx) * tx / tz + S(cam.cx);
  P.v = S(cam.fy) * ty / tz + S(cam.cy);
  P.o = S(1.0) / (S(1.0) + exp(-logit));
  // view-dependent colour
  const double cpos[3] = {-(R[0] * cam.t[0] + R[3] * cam.t[1] + R[6] * cam.t[2]),
                          -(R[1] * cam.t[0] + R[4] * cam.t[1] + R[7] * cam.t[2]),
                          -(R[2] * cam.t[0] + R[5] * cam.t[1] + R[8] * cam.t[2])};
  S dv[3] = {mu[0] - S(cpos[0]), mu[1] - S(cpos[1]), mu[2] - S(cpos[2])};
  S dn = sqrt(dv[0] * dv[0] + dv[1] * dv[1] + dv[2] * dv[2]);
  S dx = dv[0] / dn, dy = dv[1] / dn, dz = dv[2] / dn;
  for (int ch = 0; ch < 3; ++ch) P.raw[ch] = S(0.5);
  for (int l = 0; l <= deg; ++l)
    for (int m = -l; m <= l; ++m) {
      S Y = sh_basis(l, m, dx, dy, dz);
      const int idx = l * l + l + m;
      for (int ch = 0; ch < 3; ++ch) P.raw[ch] = P.raw[ch] + Y * sh[idx * 3 + ch];
    }
  for (int ch = 0; ch < 3; ++ch) P.col[ch] = (val(P.raw[ch]) < 0.0) ? S(0.0) : P.raw[ch];
}

// Tile rectangle [x0, x1) x [y0, y1) of tiles met by the square [u-r, u+r] x [v-r, v+r].
void tile_rect(double u, double v, int r, int tile, int tx, int ty, int* rect) {
  auto cl = [](long long a, long long lo, long long hi) { return std::min(std::max(a, lo), hi); };
  rect[0] = (int)cl((long long)std::floor((u - r) / tile), 0, tx);
  rect[1] = (int)cl((long long)std::floor((v - r) / tile), 0, ty);
  rect[2] = (int)cl((long long)std::floor((u + r) / tile) + 1, 0, tx);
  rect[3] = (int)cl((long long)std::floor((v + r) / tile) + 1, 0, ty);
}

unsigned depth_key_fp32(const orc_camera& cam, const double* mu) {
  // fp32 depth in the fixed evaluation order ((R6*x + R7*y) + R8*z) + t2, one rounding each
  volatile float p0 = (float)cam.R[6] * (float)mu[0];
  volatile float p1 = (float)cam.R[7] * (float)mu[1];
  volatile float p2 = (float)cam.R[8] * (float)mu[2];
  volatile float s0 = p0 + p1;
  volatile float s1 = s0 + p2;
  volatile float z = s1 + (float)cam.t[2];
  float zz = z;
  unsigned bits;
  std::memcpy(&bits, &zz, 4);
  return bits;
}

// ---------------------------------------------------------------------------------------
// Per-pixel blend.
struct Added { int id; double alpha, alpha_raw, T, sigma, gexp, dx, dy; bool clamped; };

bool toggled(const int* tg, int nt, int id, int type) {
  for (int i = 0; i < nt; ++i)
    if (tg[2 * i] == id && tg[2 * i + 1] == type) return true;
  return false;
}

void add_event(int* ev, int max_ev, int* n_ev, int id, int type) {
  if (!n_ev) return;
  if (*n_ev < max_ev && ev) { ev[2 * *n_ev] = id; ev[2 * *n_ev + 1] = type; }
  ++*n_ev;
}

// The blend of one pixel, as 3D Gaussian Splatting defines it (Section 1 by citation): front
// to back over the tile's list, sigma = 1/2 d^T conic d at the pixel centre, alpha =
// min(alpha_max, o exp(-sigma)); an entry with sigma < 0 or alpha < alpha_min is skipped; the
// pixel stops before an entry that would take T (1 - alpha) below t_min; otherwise
// C += alpha T c and T *= 1 - alpha.  Returns the contributors in order and A = (C, 1 - T).
void blend_pixel(const orc_splats* s, const int* list, int len, int px, int py,
                 const orc_opts& op, std::vector<Added>& added, double A[4], double* T_final,
                 int* n_used) {
  const double cxp = px + 0.5, cyp = py + 0.5;
  double T = 1.0, C[3] = {0, 0, 0};
  int used = 0;
  added.clear();
  for (int k = 0; k < len; ++k) {
    const int id = list[k];
    const double dx = cxp - s->uv[2 * id], dy = cyp - s->uv[2 * id + 1];
    const double ca = s->conic[3 * id], cb = s->conic[3 * id + 1], cc = s->conic[3 * id + 2];
    const double sigma = 0.5 * (ca * dx * dx + cc * dy * dy) + cb * dx * dy;
    const double ge = std::exp(-sigma);
    const double araw = s->opacity[id] * ge;
    const bool clamped = araw > op.alpha_max;
    const double alpha = clamped ? op.alpha_max : araw;
    if (sigma < 0.0 || alpha < op.alpha_min) continue;
    const double test = T * (1.0 - alpha);
    if (test < op.t_min) break;
    for (int ch = 0; ch < 3; ++ch) C[ch] += alpha * T * s->rgb[3 * id + ch];
    added.push_back(Added{id, alpha, araw, T, sigma, ge, dx, dy, clamped});
    T = test;
    used = k + 1;
  }
  A[0] = C[0]; A[1] = C[1]; A[2] = C[2]; A[3] = 1.0 - T;
  *T_final = T;
  *n_used = used;
}

// Test-harness form of blend_pixel, used only to compare an fp32 implementation with it: the
// same loop, which also reports the decisions that lie within a stated uncertainty model's
// reach of their thresholds (skip, stop, alpha clamp; mg), and takes the opposite branch of
// the decisions listed in tg (pairs of Gaussian id, event), so that every combination of the
// ambiguous decisions can be rendered.  With no toggles its result equals blend_pixel's (a
// pinned property).
void blend_pixel_probe(const orc_splats* s, const int* list, int len, int px, int py,
                       const orc_opts& op, const int* tg, int nt, const orc_margins* mg,
                       std::vector<Added>& added, double A[4], double* T_final, int* n_used,
                       int* ev, int max_ev, int* n_ev) {
  const double cxp = px + 0.5, cyp = py + 0.5;
  double T = 1.0, C[3] = {0, 0, 0};
  double epsT = 0.0;   // running relative uncertainty of T (event reporting only)
  int used = 0;
  added.clear();
  for (int k = 0; k < len; ++k) {
    const int id = list[k];
    const double u = s->uv[2 * id], v = s->uv[2 * id + 1];
    const double ca = s->conic[3 * id], cb = s->conic[3 * id + 1], cc = s->conic[3 * id + 2];
    const double dx = cxp - u, dy = cyp - v;
    const double sigma = 0.5 * (ca * dx * dx + cc * dy * dy) + cb * dx * dy;
    const double o = s->opacity[id];
    const double ge = std::exp(-sigma);
    const double araw = o * ge;
    const bool clamped = araw > op.alpha_max;
    const double alpha = clamped ? op.alpha_max : araw;
    double msig = 0.0, ma = 0.0;
    if (mg) {
      const double Sabs = 0.5 * (std::fabs(ca) * dx * dx + std::fabs(cc) * dy * dy) +
                          std::fabs(cb * dx * dy);
      const double gu = std::fabs(ca * dx + cb * dy), gv = std::fabs(cb * dx + cc * dy);
      msig = gu * mg->m_uv[2 * id] + gv * mg->m_uv[2 * id + 1] +
             (mg->m_conic[id] + mg->k_arith) * Sabs + 1e-12;
      ma = msig + mg->eps_alpha;
      if (sigma < msig) add_event(ev, max_ev, n_ev, id, ORC_EV_SKIP);
      else if (!clamped && std::fabs(araw - op.alpha_min) <= op.alpha_min * ma)
        add_event(ev, max_ev, n_ev, id, ORC_EV_SKIP);
      if (std::fabs(araw - op.alpha_max) <= op.alpha_max * ma)
        add_event(ev, max_ev, n_ev, id, ORC_EV_CLAMP);
    }
    bool skip = (sigma < 0.0) || (alpha < op.alpha_min);
    if (toggled(tg, nt, id, ORC_EV_SKIP)) skip = !skip;
    if (skip) continue;
    const double test = T * (1.0 - alpha);
    if (mg) {
      const double e = epsT + alpha / (1.0 - alpha) * ma + mg->eps_step;
      if (std::fabs(test - op.t_min) <= op.t_min * e) add_event(ev, max_ev, n_ev, id, ORC_EV_TERM);
      epsT = e;
    }
    bool stop = test < op.t_min;
    if (toggled(tg, nt, id, ORC_EV_TERM)) stop = !stop;
    if (stop) break;
    for (int ch = 0; ch < 3; ++ch) C[ch] += alpha * T * s->rgb[3 * id + ch];
    added.push_back(Added{id, alpha, araw, T, sigma, ge, dx, dy,
                          toggled(tg, nt, id, ORC_EV_CLAMP) ? !clamped : clamped});
    T = test;
    used = k + 1;
  }
  A[0] = C[0]; A[1] = C[1]; A[2] = C[2]; A[3] = 1.0 - T;
  *T_final = T;
  *n_used = used;
}

// The plain blend, or the harness form when toggles or margins are given.
void blend_any(const orc_splats* s, const int* list, int len, int px, int py,
               const orc_opts& op, const int* tg, int nt, const orc_margins* mg,
               std::vector<Added>& added, double A[4], double* T_final, int* n_used,
               int* ev, int max_ev, int* n_ev) {
  if (nt == 0 && !mg) {
    if (n_ev) *n_ev = 0;
    blend_pixel(s, list, len, px, py, op, added, A, T_final, n_used);
  } else {
    blend_pixel_probe(s, list, len, px, py, op, tg, nt, mg, added, A, T_final, n_used, ev,
                      max_ev, n_ev);
  }
}

void over(const double* X, const double* Y, double* out) {   // X over Y, premultiplied
  const double k = 1.0 - X[3];
  for (int c = 0; c < 4; ++c) out[c] = X[c] + k * Y[c];
}

void composite_out(const double A[4], const double* F, const double* B, const double* bg,
                   double out[4]) {
  const double zero[4] = {0, 0, 0, 0};
  const double* Fp = F ? F : zero;
  const double* Bp = B ? B : zero;
  double AB[4];
  over(A, Bp, AB);
  over(Fp, AB, out);
  if (bg)
    for (int c = 0; c < 3; ++c) out[c] += (1.0 - out[3]) * bg[c];
}

// 11-tap normalised Gaussian window, sigma 1.5.
void ssim_window(double w[11]) {
  double s = 0.0;
  for (int i = 0; i < 11; ++i) { w[i] = std::exp(-((i - 5.0) * (i - 5.0)) / (2.0 * 1.5 * 1.5)); s += w[i]; }
  for (int i = 0; i < 11; ++i) w[i] /= s;
}

// Direct 2-D weighted window sum with zero padding: out(p) = sum_{i,j} w_i w_j f(p + (i-5, j-5)).
void window_sum(int W, int H, const std::vector<double>& f, const double w[11],
                std::vector<double>& out) {
  out.assign((size_t)W * H, 0.0);
#pragma omp parallel for schedule(static)
  for (int y = 0; y < H; ++y)
    for (int x = 0; x < W; ++x) {
      double acc = 0.0;
      for (int i = 0; i < 11; ++i) {
        const int yy = y + i - 5;
        if (yy < 0 || yy >= H) continue;
        for (int j = 0; j < 11; ++j) {
          const int xx = x + j - 5;
          if (xx < 0 || xx >= W) continue;
          acc += w[i] * w[j] * f[(size_t)yy * W + xx];
        }
      }
      out[(size_t)y * W + x] = acc;
    }
}

}  // namespace

// =======================================================================================
extern "C" {

void orc_default_opts(orc_opts* o) {
  o->near_z = 0.2;
  o->dilation = 0.3;
  o->guard = 1.3;
  o->alpha_max = 0.99;
  o->alpha_min = 1.0 / 255.0;
  o->t_min = 1e-4;
  o->tile = 16;
}

double orc_sh_basis(int l, int m, double x, double y, double z) {
  return sh_basis<double>(l, m, x, y, z);
}

int orc_project(const orc_gaussians* g, const orc_camera* cam, const orc_opts* o,
                orc_projected* out) {
  if (!g || !cam || !o || !out || g->sh_degree < 0 || g->sh_degree > 3) return -1;
  const int D = (g->sh_degree + 1) * (g->sh_degree + 1);
  const int tx = (cam->width + o->tile - 1) / o->tile, ty = (cam->height + o->tile - 1) / o->tile;
#pragma omp parallel for schedule(static)
  for (int i = 0; i < g->n; ++i) {
    Proj<double> P;
    project_one<double>(g->means + 3 * i, g->log_scales + 3 * i, g->quats + 4 * i,
                        g->opacity_logits[i], g->sh + (size_t)i * D * 3, g->sh_degree, *cam, *o, P);
    out->depth[i] = P.tz;
    out->depth_key[i] = depth_key_fp32(*cam, g->means + 3 * i);
    int vis = P.front ? 1 : 0;
    int* rect = out->rect + 4 * i;
    rect[0] = rect[1] = rect[2] = rect[3] = 0;
    if (vis) {
      out->uv[2 * i] = P.u; out->uv[2 * i + 1] = P.v;
      out->conic[3 * i] = P.ca; out->conic[3 * i + 1] = P.cb; out->conic[3 * i + 2] = P.cc;
      out->opacity[i] = P.o;
      for (int c = 0; c < 3; ++c) { out->rgb[3 * i + c] = P.col[c]; out->rgb_raw[3 * i + c] = P.raw[c]; }
      out->eig[2 * i] = P.lam_max; out->eig[2 * i + 1] = P.lam_min;
      out->radius_exact[i] = P.r_exact;
      out->radius[i] = (int)std::ceil(P.r_exact);
      out->view_tan[2 * i] = P.tan_x; out->view_tan[2 * i + 1] = P.tan_y;
      tile_rect(P.u, P.v, out->radius[i], o->tile, tx, ty, rect);
      if (!(rect[0] < rect[2] && rect[1] < rect[3])) vis = 0;
    }
    if (!vis) {
      for (int c = 0; c < 4; ++c) rect[c] = 0;
      out->radius[i] = 0;
      if (!P.front) {
        out->uv[2 * i] = out->uv[2 * i + 1] = 0; out->opacity[i] = 0;
        for (int c = 0; c < 3; ++c) { out->conic[3 * i + c] = 0; out->rgb[3 * i + c] = 0; out->rgb_raw[3 * i + c] = 0; }
        out->eig[2 * i] = out->eig[2 * i + 1] = 0; out->radius_exact[i] = 0;
        out->view_tan[2 * i] = out->view_tan[2 * i + 1] = 0;
      }
    }
    out->visible[i] = vis;
  }
  return 0;
}

int orc_project_backward(const orc_gaussians* g, const orc_camera* cam, const orc_opts* o,
                         const double* grad2d, double* d_means, double* d_log_scales,
                         double* d_quats, double* d_opacity_logits, double* d_sh) {
  if (!g || g->sh_degree < 0 || g->sh_degree > 3) return -1;
  const int D = (g->sh_degree + 1) * (g->sh_degree + 1);
  const int tx = (cam->width + o->tile - 1) / o->tile, ty = (cam->height + o->tile - 1) / o->tile;
#pragma omp parallel for schedule(dynamic, 16)
  for (int i = 0; i < g->n; ++i) {
    // seed tangents: mean 0-2, log-scale 3-5, quat 6-9, logit 10, sh 11..
    Dual mu[3], ls[3], q[4], lg, sh[48];
    for (int k = 0; k < 3; ++k) { mu[k] = Dual(g->means[3 * i + k]); mu[k].d[k] = 1.0; }
    for (int k = 0; k < 3; ++k) { ls[k] = Dual(g->log_scales[3 * i + k]); ls[k].d[3 + k] = 1.0; }
    for (int k = 0; k < 4; ++k) { q[k] = Dual(g->quats[4 * i + k]); q[k].d[6 + k] = 1.0; }
    lg = Dual(g->opacity_logits[i]); lg.d[10] = 1.0;
    for (int k = 0; k < D * 3; ++k) { sh[k] = Dual(g->sh[(size_t)i * D * 3 + k]); sh[k].d[11 + k] = 1.0; }
    Proj<Dual> P;
    project_one<Dual>(mu, ls, q, lg, sh, g->sh_degree, *cam, *o, P);
    double grad[NT] = {0};
    bool vis = P.front;
    if (vis) {
      int rect[4];
      tile_rect(P.u.v, P.v.v, (int)std::ceil(P.r_exact), o->tile, tx, ty, rect);
      vis = rect[0] < rect[2] && rect[1] < rect[3];
    }
    if (vis) {
      const Dual* outs[9] = {&P.u, &P.v, &P.ca, &P.cb, &P.cc, &P.o, &P.col[0], &P.col[1], &P.col[2]};
      for (int k = 0; k < 9; ++k) {
        const double gk = grad2d[9 * i + k];
        for (int j = 0; j < NT; ++j) grad[j] += gk * outs[k]->d[j];
      }
    }
    for (int k = 0; k < 3; ++k) d_means[3 * i + k] = grad[k];
    for (int k = 0; k < 3; ++k) d_log_scales[3 * i + k] = grad[3 + k];
    for (int k = 0; k < 4; ++k) d_quats[4 * i + k] = grad[6 + k];
    d_opacity_logits[i] = grad[10];
    for (int k = 0; k < D * 3; ++k) d_sh[(size_t)i * D * 3 + k] = grad[11 + k];
  }
  return 0;
}

double orc_box_min_sigma(const double* q, double X0, double X1, double Y0, double Y1) {
  if (X0 <= 0.0 && X1 >= 0.0 && Y0 <= 0.0 && Y1 >= 0.0) return 0.0;
  auto sig = [q](double dx, double dy) { return 0.5 * (q[0] * dx * dx + q[2] * dy * dy) + q[1] * dx * dy; };
  double best = HUGE_VAL;
  for (double X : {X0, X1}) {          // edge dx = X: d sigma / d dy = b X + c dy = 0
    const double dy = std::min(std::max(-q[1] * X / q[2], Y0), Y1);
    best = std::min(best, sig(X, dy));
  }
  for (double Y : {Y0, Y1}) {          // edge dy = Y: a dx + b Y = 0
    const double dx = std::min(std::max(-q[1] * Y / q[0], X0), X1);
    best = std::min(best, sig(dx, Y));
  }
  return best;
}

long long orc_tile_lists(int n, const int* visible, const int* rect, const unsigned* depth_key,
                         int tiles_x, int tiles_y, long long* offsets, int* ids,
                         long long capacity, const orc_splats* s, double alpha_min, int tile,
                         double margin_rel, double margin_abs) {
  struct Item { long long tile; unsigned key; int id; };
  std::vector<Item> items;
  for (int i = 0; i < n; ++i) {
    if (!visible[i]) continue;
    const int* r = rect + 4 * i;
    for (int y = r[1]; y < r[3]; ++y)
      for (int x = r[0]; x < r[2]; ++x) {
        if (s) {
          const double o = s->opacity[i];
          if (!(o >= alpha_min)) continue;
          const double u = s->uv[2 * i], v = s->uv[2 * i + 1];
          const double m = orc_box_min_sigma(s->conic + 3 * i, x * tile + 0.5 - u,
                                             x * tile + tile - 0.5 - u, y * tile + 0.5 - v,
                                             y * tile + tile - 0.5 - v);
          // keep when m <= ln(o / alpha_min) (the Gaussian reaches alpha_min somewhere on the
          // tile), or, with a margin, when m log2(e) <= (thr (1 + rel) + abs) (1 + rel) with
          // thr = log2(o / alpha_min): a superset whose extra entries no pixel of t reaches
          const double thr2 = std::log2(o / alpha_min);
          const double lim2 = (thr2 * (1.0 + margin_rel) + margin_abs) * (1.0 + margin_rel);
          if (margin_rel == 0.0 && margin_abs == 0.0) {
            if (m > std::log(o / alpha_min)) continue;
          } else if (m / std::log(2.0) > lim2) {
            continue;
          }
        }
        items.push_back(Item{(long long)y * tiles_x + x, depth_key[i], i});
      }
  }
  std::stable_sort(items.begin(), items.end(), [](const Item& a, const Item& b) {
    if (a.tile != b.tile) return a.tile < b.tile;
    return a.key < b.key;
  });
  const long long K = (long long)items.size();
  if (K > capacity) return -K - 1;
  const long long nt = (long long)tiles_x * tiles_y;
  for (long long t = 0; t <= nt; ++t) offsets[t] = 0;
  for (const Item& it : items) offsets[it.tile + 1]++;
  for (long long t = 0; t < nt; ++t) offsets[t + 1] += offsets[t];
  for (long long k = 0; k < K; ++k) ids[k] = items[k].id;
  return K;
}

int orc_render_pixel(const orc_splats* s, const int* list, int len, int px, int py,
                     const orc_opts* o, const double* F, const double* B, const double* bg,
                     const int* toggles, int n_toggles, const orc_margins* mg,
                     double* out4, double* A4, double* T_final, int* n_used,
                     int* ev, int max_ev, int* n_ev) {
  std::vector<Added> added;
  if (n_ev) *n_ev = 0;
  blend_any(s, list, len, px, py, *o, toggles, n_toggles, mg, added, A4, T_final, n_used,
              ev, max_ev, n_ev);
  composite_out(A4, F, B, bg, out4);
  return 0;
}

int orc_render_image(const orc_splats* s, const long long* offsets, const int* ids,
                     int width, int height, const orc_opts* o, const double* F,
                     const double* B, const double* bg, const orc_margins* mg,
                     double* out, double* A, double* T_final, int* n_used,
                     int* ev, int max_ev, int* n_ev) {
  const int tx = (width + o->tile - 1) / o->tile;
#pragma omp parallel for schedule(dynamic, 64)
  for (int p = 0; p < width * height; ++p) {
    const int px = p % width, py = p / width;
    const long long t = (long long)(py / o->tile) * tx + (px / o->tile);
    const long long b = offsets[t], e = offsets[t + 1];
    std::vector<Added> added;
    double A4[4], o4[4], Tf;
    int nu, ne = 0;
    blend_any(s, ids + b, (int)(e - b), px, py, *o, nullptr, 0, mg, added, A4, &Tf, &nu,
                ev ? ev + (size_t)p * max_ev * 2 : nullptr, max_ev, n_ev ? &ne : nullptr);
    composite_out(A4, F ? F + 4 * (size_t)p : nullptr, B ? B + 4 * (size_t)p : nullptr, bg, o4);
    for (int c = 0; c < 4; ++c) {
      if (out) out[4 * (size_t)p + c] = o4[c];
      if (A) A[4 * (size_t)p + c] = A4[c];
    }
    if (T_final) T_final[p] = Tf;
    if (n_used) n_used[p] = nu;
    if (n_ev) n_ev[p] = ne;
  }
  return 0;
}

int orc_backward_pixel(const orc_splats* s, const int* list, int len, int px, int py,
                       const orc_opts* o, const double* F, const double* B, const double* bg,
                       const int* toggles, int n_toggles, const double* G, double* grad2d) {
  std::vector<Added> added;
  double A[4], Tf;
  int nu;
  blend_any(s, list, len, px, py, *o, toggles, n_toggles, nullptr, added, A, &Tf, &nu,
              nullptr, 0, nullptr);
  // d final / d A: out = F over (A over B), final.rgb = out.rgb + (1 - out.a) bg
  const double Fa = F ? F[3] : 0.0;
  const double Brgb[3] = {B ? B[0] : 0.0, B ? B[1] : 0.0, B ? B[2] : 0.0};
  const double Ba = B ? B[3] : 0.0;
  double Grgb[3], Ga = 0.0;
  for (int c = 0; c < 3; ++c) Grgb[c] = (1.0 - Fa) * G[c];
  for (int c = 0; c < 3; ++c) Ga -= (1.0 - Fa) * G[c] * Brgb[c];
  if (bg)
    for (int c = 0; c < 3; ++c) Ga -= (1.0 - Fa) * (1.0 - Ba) * G[c] * bg[c];
  // back to front: R = colour accumulated behind the current Gaussian
  double Rc[3] = {0, 0, 0};
  for (int i = (int)added.size() - 1; i >= 0; --i) {
    const Added& a = added[i];
    const double* col = s->rgb + 3 * a.id;
    double dalpha = Ga * Tf / (1.0 - a.alpha);
    for (int c = 0; c < 3; ++c) dalpha += Grgb[c] * (a.T * col[c] - Rc[c] / (1.0 - a.alpha));
    double* gr = grad2d + 9 * (size_t)a.id;
    for (int c = 0; c < 3; ++c) gr[6 + c] += Grgb[c] * a.alpha * a.T;
    for (int c = 0; c < 3; ++c) Rc[c] += a.alpha * a.T * col[c];
    if (a.clamped) continue;   // d min(alpha_max, .) = 0 on the clamped side
    // alpha = o exp(-sigma)
    const double o_ = s->opacity[a.id];
    gr[5] += dalpha * a.gexp;
    const double dsig = -dalpha * o_ * a.gexp;
    const double ca = s->conic[3 * a.id], cb = s->conic[3 * a.id + 1], cc = s->conic[3 * a.id + 2];
    // sigma = 0.5 (ca dx^2 + cc dy^2) + cb dx dy, dx = px + 0.5 - u
    gr[0] += dsig * -(ca * a.dx + cb * a.dy);
    gr[1] += dsig * -(cb * a.dx + cc * a.dy);
    gr[2] += dsig * 0.5 * a.dx * a.dx;
    gr[3] += dsig * a.dx * a.dy;
    gr[4] += dsig * 0.5 * a.dy * a.dy;
  }
  return 0;
}

int orc_backward_image(const orc_splats* s, const long long* offsets, const int* ids,
                       int width, int height, const orc_opts* o, const double* F,
                       const double* B, const double* bg, const double* G, double* grad2d) {
  const int tx = (width + o->tile - 1) / o->tile;
  std::memset(grad2d, 0, sizeof(double) * 9 * (size_t)s->n);
  for (int p = 0; p < width * height; ++p) {   // serial: per-Gaussian sums in pixel order
    const int px = p % width, py = p / width;
    const long long t = (long long)(py / o->tile) * tx + (px / o->tile);
    orc_backward_pixel(s, ids + offsets[t], (int)(offsets[t + 1] - offsets[t]), px, py, o,
                       F ? F + 4 * (size_t)p : nullptr, B ? B + 4 * (size_t)p : nullptr, bg,
                       nullptr, 0, G + 3 * (size_t)p, grad2d);
  }
  return 0;
}

int orc_backward_pixels(const orc_splats* s, const long long* offsets, const int* ids,
                        int width, int height, const orc_opts* o, const double* F,
                        const double* B, const double* bg, const double* G,
                        const int* pixels, int n_pixels, double* grad2d) {
  // the same sum as orc_backward_image over the listed pixels only: a pixel whose upstream
  // gradient G is zero adds exactly zero to every component, so for a G that vanishes
  // outside the list the two agree
  const int tx = (width + o->tile - 1) / o->tile;
  std::memset(grad2d, 0, sizeof(double) * 9 * (size_t)s->n);
  for (int k = 0; k < n_pixels; ++k) {
    const int p = pixels[k];
    if (p < 0 || p >= width * height) return 1;
    const int px = p % width, py = p / width;
    const long long t = (long long)(py / o->tile) * tx + (px / o->tile);
    orc_backward_pixel(s, ids + offsets[t], (int)(offsets[t + 1] - offsets[t]), px, py, o,
                       F ? F + 4 * (size_t)p : nullptr, B ? B + 4 * (size_t)p : nullptr, bg,
                       nullptr, 0, G + 3 * (size_t)p, grad2d);
  }
  return 0;
}

int orc_composite_layers(int n_pixels, const double* layers, const int* order, int count,
                         double* out) {
#pragma omp parallel for schedule(static)
  for (int p = 0; p < n_pixels; ++p) {
    double acc[4] = {0, 0, 0, 0}, nxt[4];
    for (int k = 0; k < count; ++k) {
      over(acc, layers + ((size_t)order[k] * n_pixels + p) * 4, nxt);
      for (int c = 0; c < 4; ++c) acc[c] = nxt[c];
    }
    for (int c = 0; c < 4; ++c) out[4 * (size_t)p + c] = acc[c];
  }
  return 0;
}

int orc_layer_visibility(int n_pixels, int n_layers, const double* layers, const int* order,
                         int count, double* visible, double* coverage) {
  std::vector<char> seen(n_layers > 0 ? n_layers : 0, 0);
  for (int k = 0; k < count; ++k) {
    if (order[k] < 0 || order[k] >= n_layers || seen[order[k]]) return 1;
    seen[order[k]] = 1;
  }
  std::vector<double> vis(n_layers > 0 ? n_layers : 0, 0.0), cov(vis);
  for (int p = 0; p < n_pixels; ++p) {
    double T = 1.0;                  // product of (1 - alpha) over the layers walked so far
    for (int k = 0; k < count; ++k) {
      const int j = order[k];
      const double a = layers[((size_t)j * n_pixels + p) * 4 + 3];
      vis[j] += a * T;
      cov[j] += a;
      T *= 1.0 - a;
    }
  }
  for (int j = 0; j < n_layers; ++j) {
    visible[j] = vis[j] / n_pixels;
    coverage[j] = cov[j] / n_pixels;
  }
  return 0;
}

int orc_ssim_map(int width, int height, const double* x, const double* y, double* map) {
  const double C1 = 0.01 * 0.01, C2 = 0.03 * 0.03;
  double w[11];
  ssim_window(w);
  const size_t P = (size_t)width * height;
  std::vector<double> xc(P), yc(P), xx(P), yy(P), xy(P), mx, my, sxx, syy, sxy;
  for (int ch = 0; ch < 3; ++ch) {
    for (size_t p = 0; p < P; ++p) {
      xc[p] = x[3 * p + ch]; yc[p] = y[3 * p + ch];
      xx[p] = xc[p] * xc[p]; yy[p] = yc[p] * yc[p]; xy[p] = xc[p] * yc[p];
    }
    window_sum(width, height, xc, w, mx);
    window_sum(width, height, yc, w, my);
    window_sum(width, height, xx, w, sxx);
    window_sum(width, height, yy, w, syy);
    window_sum(width, height, xy, w, sxy);
    for (size_t p = 0; p < P; ++p) {
      const double vx = sxx[p] - mx[p] * mx[p], vy = syy[p] - my[p] * my[p];
      const double cxy = sxy[p] - mx[p] * my[p];
      map[3 * p + ch] = ((2 * mx[p] * my[p] + C1) * (2 * cxy + C2)) /
                        ((mx[p] * mx[p] + my[p] * my[p] + C1) * (vx + vy + C2));
    }
  }
  return 0;
}

int orc_loss(int width, int height, const double* x, const double* y, double lam,
             double* loss, double* grad) {
  const double C1 = 0.01 * 0.01, C2 = 0.03 * 0.03;
  const size_t P = (size_t)width * height;
  const double inv = 1.0 / (3.0 * (double)P);
  double l1 = 0.0, ssim = 0.0;
  for (size_t k = 0; k < 3 * P; ++k) l1 += std::fabs(x[k] - y[k]);
  if (grad)
    for (size_t k = 0; k < 3 * P; ++k) {
      const double d = x[k] - y[k];
      grad[k] = (1.0 - lam) * inv * ((d > 0) - (d < 0));
    }
  double w[11];
  ssim_window(w);
  std::vector<double> xc(P), yc(P), xx(P), yy(P), xy(P), mx, my, sxx, syy, sxy;
  std::vector<double> Am(P), Bm(P), Cm(P), wA, wB, wC;
  for (int ch = 0; ch < 3; ++ch) {
    for (size_t p = 0; p < P; ++p) {
      xc[p] = x[3 * p + ch]; yc[p] = y[3 * p + ch];
      xx[p] = xc[p] * xc[p]; yy[p] = yc[p] * yc[p]; xy[p] = xc[p] * yc[p];
    }
    window_sum(width, height, xc, w, mx);
    window_sum(width, height, yc, w, my);
    window_sum(width, height, xx, w, sxx);
    window_sum(width, height, yy, w, syy);
    window_sum(width, height, xy, w, sxy);
    for (size_t p = 0; p < P; ++p) {
      const double vx = sxx[p] - mx[p] * mx[p], vy = syy[p] - my[p] * my[p];
      const double cxy = sxy[p] - mx[p] * my[p];
      const double N1 = 2 * mx[p] * my[p] + C1, N2 = 2 * cxy + C2;
      const double D1 = mx[p] * mx[p] + my[p] * my[p] + C1, D2 = vx + vy + C2;
      const double Sv = (N1 * N2) / (D1 * D2);
      ssim += Sv;
      // partial derivatives of S w.r.t. mu_x, sigma_xx, sigma_xy at p
      const double dS_dmx = (2 * my[p] * N2 - Sv * 2 * mx[p] * D2) / (D1 * D2);
      const double dS_dvx = -Sv / D2;
      const double dS_dcxy = 2 * N1 / (D1 * D2);
      Am[p] = dS_dmx - 2 * mx[p] * dS_dvx - my[p] * dS_dcxy;
      Bm[p] = dS_dvx;
      Cm[p] = dS_dcxy;
    }
    if (grad) {
      window_sum(width, height, Am, w, wA);   // symmetric window: adjoint = same sum
      window_sum(width, height, Bm, w, wB);
      window_sum(width, height, Cm, w, wC);
      for (size_t p = 0; p < P; ++p) {
        const double dS = wA[p] + 2 * xc[p] * wB[p] + yc[p] * wC[p];
        grad[3 * p + ch] += -lam * inv * dS;
      }
    }
  }
  *loss = (1.0 - lam) * l1 * inv + lam * (1.0 - ssim * inv);
  return 0;
}

int orc_adam(long long n, double* theta, const double* grad, double* m, double* v, double lr,
             double beta1, double beta2, double eps, int step) {
  const double bc1 = 1.0 - std::pow(beta1, step), bc2 = 1.0 - std::pow(beta2, step);
  for (long long i = 0; i < n; ++i) {
    m[i] = beta1 * m[i] + (1.0 - beta1) * grad[i];
    v[i] = beta2 * v[i] + (1.0 - beta2) * grad[i] * grad[i];
    const double mh = m[i] / bc1, vh = v[i] / bc2;
    theta[i] -= lr * mh / (std::sqrt(vh) + eps);
  }
  return 0;
}

int orc_assign_cells(int n, const double* means, const double* origin, double side,
                     const int* dims, int* cell) {
  for (int i = 0; i < n; ++i) {
    int c[3];
    for (int k = 0; k < 3; ++k) {
      long long f = (long long)std::floor((means[3 * i + k] - origin[k]) / side);
      c[k] = (int)std::min<long long>(std::max<long long>(f, 0), dims[k] - 1);
    }
    cell[i] = c[0] + dims[0] * (c[1] + dims[1] * c[2]);
  }
  return 0;
}

int orc_partition_split(const int* dims, const double* origin, double side,
                        const double* campos, int active, int* front, int* nf, int* back,
                        int* nb) {
  const int n = dims[0] * dims[1] * dims[2];
  if (active < 0 || active >= n) return -1;
  long long cc[3];
  for (int k = 0; k < 3; ++k) cc[k] = (long long)std::floor((campos[k] - origin[k]) / side);
  std::vector<std::pair<long long, int>> keyed;
  long long key_a = 0;
  for (int j = 0; j < n; ++j) {
    const long long idx[3] = {j % dims[0], (j / dims[0]) % dims[1], j / (dims[0] * dims[1])};
    long long key = 0;
    for (int k = 0; k < 3; ++k) key += std::llabs(idx[k] - cc[k]);
    if (j == active) key_a = key;
    keyed.push_back({key, j});
  }
  std::sort(keyed.begin(), keyed.end());
  *nf = 0; *nb = 0;
  for (const auto& kj : keyed) {
    if (kj.second == active) continue;
    if (kj.first < key_a) front[(*nf)++] = kj.second;
    else back[(*nb)++] = kj.second;
  }
  return 0;
}

}  // extern "C"

// ---------------------------------------------------------------------------------------
// Visible camera-partition pairs (Section 2: the visible pairs are cached; Section 3: the
// cameras left after frustum filtering).

int orc_block_bounds(const orc_gaussians* g, double* box) {
  for (int k = 0; k < 3; ++k) { box[k] = HUGE_VAL; box[3 + k] = -HUGE_VAL; }
  for (int i = 0; i < g->n; ++i) {
    const double* q = g->quats + 4 * i;
    const double qn = std::sqrt(q[0] * q[0] + q[1] * q[1] + q[2] * q[2] + q[3] * q[3]);
    const double w = q[0] / qn, x = q[1] / qn, y = q[2] / qn, z = q[3] / qn;
    const double R[3][3] = {{1 - 2 * (y * y + z * z), 2 * (x * y - w * z), 2 * (x * z + w * y)},
                            {2 * (x * y + w * z), 1 - 2 * (x * x + z * z), 2 * (y * z - w * x)},
                            {2 * (x * z - w * y), 2 * (y * z + w * x), 1 - 2 * (x * x + y * y)}};
    double S2[3];
    for (int j = 0; j < 3; ++j) S2[j] = std::exp(2.0 * g->log_scales[3 * i + j]);
    for (int k = 0; k < 3; ++k) {
      // Sigma_kk = sum_j R_kj^2 s_j^2: the ellipsoid's half-width along axis k is 3 sqrt(Sigma_kk)
      double v = 0.0;
      for (int j = 0; j < 3; ++j) v += R[k][j] * R[k][j] * S2[j];
      const double e = 3.0 * std::sqrt(v), m = g->means[3 * i + k];
      box[k] = std::min(box[k], m - e);
      box[3 + k] = std::max(box[3 + k], m + e);
    }
  }
  return 0;
}

int orc_pair_visible(const orc_camera* cam, const orc_opts* o, const double* box, int* visible) {
  if (!(box[0] <= box[3] && box[1] <= box[4] && box[2] <= box[5])) { *visible = 0; return 0; }
  const double gx = o->guard * 0.5 * cam->width / cam->fx;
  const double gy = o->guard * 0.5 * cam->height / cam->fy;
  // the box's eight corners in camera space
  double pc[8][3];
  for (int c = 0; c < 8; ++c) {
    const double p[3] = {box[(c & 1) ? 3 : 0], box[(c & 2) ? 4 : 1], box[(c & 4) ? 5 : 2]};
    for (int i = 0; i < 3; ++i) {
      pc[c][i] = cam->t[i];
      for (int j = 0; j < 3; ++j) pc[c][i] += cam->R[3 * i + j] * p[j];
    }
  }
  // culled when all corners lie outside one bounding plane of the frustum (a linear function
  // is largest over the box at a corner)
  auto all_out = [&](auto outside) {
    for (int c = 0; c < 8; ++c)
      if (!outside(pc[c][0], pc[c][1], pc[c][2])) return false;
    return true;
  };
  const bool culled =
      all_out([&](double, double, double z) { return z < o->near_z; }) ||
      all_out([&](double x, double, double z) { return x > gx * z; }) ||
      all_out([&](double x, double, double z) { return -x > gx * z; }) ||
      all_out([&](double, double y, double z) { return y > gy * z; }) ||
      all_out([&](double, double y, double z) { return -y > gy * z; });
  *visible = culled ? 0 : 1;
  return 0;
}
