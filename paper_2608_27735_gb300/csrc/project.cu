// K2 (projection) and K8 (projection backward) of the ABCD active-block step.
//
// 3D Gaussian Splatting's EWA projection (the renderer the paper instantiates, Section 1):
// t = W mu + t_cam; Sigma = R(q) S S^T R(q)^T; Sigma' = J W Sigma W^T J^T + dilation*I with
// J the perspective Jacobian at the (guarded) mean; conic = Sigma'^-1; radius = ceil(3 sqrt
// lambda_max); colour = real SH at the view direction + 0.5, clamped at 0; opacity =
// sigmoid(logit).  One thread per Gaussian; the block is small (<= a few 1e5 Gaussians).
#include "abcd_internal.cuh"

namespace abcd {
namespace {

struct Params {            // active-block parameters (device SoA)
  const float* means;
  const float* log_scales;
  const float* quats;
  const float* logits;
  const float* sh;
};

// Real SH basis at unit direction (x, y, z), degree <= deg, and optionally its Cartesian
// gradient.  Y = k[i] * (d^m P_l / dz^m)(z) * Re/Im (x + i y)^m with the Legendre
// polynomials P1 = z, P2 = (3z^2 - 1)/2, P3 = (5z^3 - 3z)/2.
__device__ __forceinline__ void sh_eval(const SHConst& K, int deg, float x, float y, float z,
                                        float* Y, float (*dY)[3]) {
  Y[0] = K.k[0];
  if (dY) { dY[0][0] = dY[0][1] = dY[0][2] = 0.f; }
  if (deg < 1) return;
  Y[1] = K.k[1] * y;
  Y[2] = K.k[2] * z;
  Y[3] = K.k[3] * x;
  if (dY) {
    dY[1][0] = 0.f; dY[1][1] = K.k[1]; dY[1][2] = 0.f;
    dY[2][0] = 0.f; dY[2][1] = 0.f; dY[2][2] = K.k[2];
    dY[3][0] = K.k[3]; dY[3][1] = 0.f; dY[3][2] = 0.f;
  }
  if (deg < 2) return;
  const float xx = x * x, yy = y * y, zz = z * z;
  Y[4] = K.k[4] * 6.f * x * y;                 // P2'' = 3, Im (x+iy)^2 = 2xy
  Y[5] = K.k[5] * 3.f * z * y;                 // P2' = 3z
  Y[6] = K.k[6] * (1.5f * zz - 0.5f);
  Y[7] = K.k[7] * 3.f * z * x;
  Y[8] = K.k[8] * 3.f * (xx - yy);             // Re (x+iy)^2 = x^2 - y^2
  if (dY) {
    dY[4][0] = K.k[4] * 6.f * y; dY[4][1] = K.k[4] * 6.f * x; dY[4][2] = 0.f;
    dY[5][0] = 0.f; dY[5][1] = K.k[5] * 3.f * z; dY[5][2] = K.k[5] * 3.f * y;
    dY[6][0] = 0.f; dY[6][1] = 0.f; dY[6][2] = K.k[6] * 3.f * z;
    dY[7][0] = K.k[7] * 3.f * z; dY[7][1] = 0.f; dY[7][2] = K.k[7] * 3.f * x;
    dY[8][0] = K.k[8] * 6.f * x; dY[8][1] = -K.k[8] * 6.f * y; dY[8][2] = 0.f;
  }
  if (deg < 3) return;
  const float p3d1 = 7.5f * zz - 1.5f;         // P3' = (15 z^2 - 3)/2
  Y[9] = K.k[9] * 15.f * (3.f * xx * y - yy * y);      // P3''' = 15, Im (x+iy)^3
  Y[10] = K.k[10] * 30.f * z * x * y;                  // P3'' = 15 z, Im (x+iy)^2 = 2xy
  Y[11] = K.k[11] * p3d1 * y;
  Y[12] = K.k[12] * (2.5f * zz * z - 1.5f * z);
  Y[13] = K.k[13] * p3d1 * x;
  Y[14] = K.k[14] * 15.f * z * (xx - yy);
  Y[15] = K.k[15] * 15.f * (xx * x - 3.f * x * yy);    // Re (x+iy)^3
  if (dY) {
    dY[9][0] = K.k[9] * 90.f * x * y; dY[9][1] = K.k[9] * 45.f * (xx - yy); dY[9][2] = 0.f;
    dY[10][0] = K.k[10] * 30.f * z * y; dY[10][1] = K.k[10] * 30.f * z * x; dY[10][2] = K.k[10] * 30.f * x * y;
    dY[11][0] = 0.f; dY[11][1] = K.k[11] * p3d1; dY[11][2] = K.k[11] * 15.f * z * y;
    dY[12][0] = 0.f; dY[12][1] = 0.f; dY[12][2] = K.k[12] * p3d1;
    dY[13][0] = K.k[13] * p3d1; dY[13][1] = 0.f; dY[13][2] = K.k[13] * 15.f * z * x;
    dY[14][0] = K.k[14] * 30.f * z * x; dY[14][1] = -K.k[14] * 30.f * z * y; dY[14][2] = K.k[14] * 15.f * (xx - yy);
    dY[15][0] = K.k[15] * 45.f * (xx - yy); dY[15][1] = -K.k[15] * 90.f * x * y; dY[15][2] = 0.f;
  }
}

// Depth along the view axis in the fixed order ((R6 x + R7 y) + R8 z) + t2, each operation
// rounded once (no contraction): this value is the sort key.
__device__ __forceinline__ float view_depth(const Cam& c, float x, float y, float z) {
  return __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(c.R[6], x), __fmul_rn(c.R[7], y)),
                             __fmul_rn(c.R[8], z)), c.t[2]);
}

struct Geo {               // forward intermediates shared by the two kernels
  float tx, ty, tz;
  float s[3];
  float qw, qx, qy, qz, qinv;
  float Rq[3][3];
  float M[3][3];
  float J00, J02, J11, J12;
  bool clx, cly;
  float T[2][3];
  float P[2][3];
  float a, b, c, det;
};

__device__ __forceinline__ void geometry(const Cam& cam, const Opts& op, const Params& p, int i,
                                         float tz, Geo& G) {
  const float mx = p.means[3 * i], my = p.means[3 * i + 1], mz = p.means[3 * i + 2];
  G.tx = cam.R[0] * mx + cam.R[1] * my + cam.R[2] * mz + cam.t[0];
  G.ty = cam.R[3] * mx + cam.R[4] * my + cam.R[5] * mz + cam.t[1];
  G.tz = tz;
  for (int k = 0; k < 3; ++k) G.s[k] = expf(p.log_scales[3 * i + k]);
  const float4 q = *reinterpret_cast<const float4*>(p.quats + 4 * (size_t)i);
  const float qn = sqrtf(q.x * q.x + q.y * q.y + q.z * q.z + q.w * q.w);
  G.qinv = 1.f / qn;
  const float w = q.x * G.qinv, x = q.y * G.qinv, y = q.z * G.qinv, z = q.w * G.qinv;
  G.qw = w; G.qx = x; G.qy = y; G.qz = z;
  G.Rq[0][0] = 1.f - 2.f * (y * y + z * z); G.Rq[0][1] = 2.f * (x * y - w * z); G.Rq[0][2] = 2.f * (x * z + w * y);
  G.Rq[1][0] = 2.f * (x * y + w * z); G.Rq[1][1] = 1.f - 2.f * (x * x + z * z); G.Rq[1][2] = 2.f * (y * z - w * x);
  G.Rq[2][0] = 2.f * (x * z - w * y); G.Rq[2][1] = 2.f * (y * z + w * x); G.Rq[2][2] = 1.f - 2.f * (x * x + y * y);
  for (int r = 0; r < 3; ++r)
    for (int k = 0; k < 3; ++k) G.M[r][k] = G.Rq[r][k] * G.s[k];
  const float itz = 1.f / tz;
  const float rx = G.tx * itz, ry = G.ty * itz;
  G.clx = rx < -cam.limx || rx > cam.limx;
  G.cly = ry < -cam.limy || ry > cam.limy;
  const float xg = fminf(fmaxf(rx, -cam.limx), cam.limx) * tz;
  const float yg = fminf(fmaxf(ry, -cam.limy), cam.limy) * tz;
  G.J00 = cam.fx * itz;
  G.J11 = cam.fy * itz;
  G.J02 = -cam.fx * xg * itz * itz;
  G.J12 = -cam.fy * yg * itz * itz;
  for (int k = 0; k < 3; ++k) {
    G.T[0][k] = G.J00 * cam.R[k] + G.J02 * cam.R[6 + k];
    G.T[1][k] = G.J11 * cam.R[3 + k] + G.J12 * cam.R[6 + k];
  }
  for (int r = 0; r < 2; ++r)
    for (int k = 0; k < 3; ++k)
      G.P[r][k] = G.T[r][0] * G.M[0][k] + G.T[r][1] * G.M[1][k] + G.T[r][2] * G.M[2][k];
  // 2-D covariance P P^T + dilation I; its determinant via Lagrange's identity
  // |p0|^2 |p1|^2 - (p0.p1)^2 = |p0 x p1|^2 (no cancellation), plus the dilation terms.
  const float a0 = G.P[0][0] * G.P[0][0] + G.P[0][1] * G.P[0][1] + G.P[0][2] * G.P[0][2];
  const float c0 = G.P[1][0] * G.P[1][0] + G.P[1][1] * G.P[1][1] + G.P[1][2] * G.P[1][2];
  G.b = G.P[0][0] * G.P[1][0] + G.P[0][1] * G.P[1][1] + G.P[0][2] * G.P[1][2];
  const float cx = G.P[0][1] * G.P[1][2] - G.P[0][2] * G.P[1][1];
  const float cy = G.P[0][2] * G.P[1][0] - G.P[0][0] * G.P[1][2];
  const float cz = G.P[0][0] * G.P[1][1] - G.P[0][1] * G.P[1][0];
  G.a = a0 + op.dilation;
  G.c = c0 + op.dilation;
  G.det = (cx * cx + cy * cy + cz * cz) + op.dilation * (a0 + c0) + op.dilation * op.dilation;
}

// SH coefficients of a warp's 32 consecutive Gaussians form one contiguous block of 32 x 3D
// floats ([n][D][3] layout); it goes through shared memory (row pitch 3D + 1, so a lane's row
// reads are conflict-free) so that the global reads and writes are coalesced.
template <int DEG>
struct ShLayout {
  static constexpr int D = (DEG + 1) * (DEG + 1);
  static constexpr int N = 3 * D;        // floats per Gaussian
  static constexpr int P = N + 1;        // shared-memory row pitch
};

template <int DEG>
__device__ __forceinline__ void sh_to_shared(const float* sh, int n, int first, float* buf) {
  constexpr int N = ShLayout<DEG>::N, P = ShLayout<DEG>::P;
  const int lane = threadIdx.x & 31;
  const int cnt = min(32, n - first);
  const float* src = sh + (size_t)first * N;
  for (int j = lane; j < cnt * N; j += 32) buf[(j / N) * P + (j % N)] = src[j];
  __syncwarp();
}

template <int DEG>
__device__ __forceinline__ void sh_from_shared(float* sh, int n, int first, const float* buf) {
  constexpr int N = ShLayout<DEG>::N, P = ShLayout<DEG>::P;
  const int lane = threadIdx.x & 31;
  const int cnt = min(32, n - first);
  float* dst = sh + (size_t)first * N;
  __syncwarp();
  for (int j = lane; j < cnt * N; j += 32) dst[j] = buf[(j / N) * P + (j % N)];
}

constexpr int kProjThreads = 128;

template <int DEG>
__global__ void __launch_bounds__(kProjThreads)
project_fwd_kernel(Params p, int n, Cam cam, Opts op, SHConst K, float2* uv,
                   float4* conic_op, float* rgb, float* depth, int* radius,
                   unsigned* tiles_touched) {
  pdl_prologue();
  constexpr int D = ShLayout<DEG>::D, P = ShLayout<DEG>::P;
  __shared__ float s_sh[kProjThreads / 32][32 * P];
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31, first = i - lane;
  if (first >= n) return;                                  // whole warp
  float* buf = s_sh[threadIdx.x >> 5];
  sh_to_shared<DEG>(p.sh, n, first, buf);
  if (i >= n) return;
  const float tz = view_depth(cam, p.means[3 * i], p.means[3 * i + 1], p.means[3 * i + 2]);
  depth[i] = tz;
  int r = 0;
  unsigned touched = 0;
  float2 uvo = make_float2(0.f, 0.f);
  float4 co = make_float4(0.f, 0.f, 0.f, 0.f);
  float col[3] = {0.f, 0.f, 0.f};
  if (tz > op.near_z) {
    Geo G;
    geometry(cam, op, p, i, tz, G);
    const float idet = 1.f / G.det;
    const float mid = 0.5f * (G.a + G.c);
    const float hd = 0.5f * (G.a - G.c);
    const float lam = mid + sqrtf(fmaxf(0.1f, hd * hd + G.b * G.b));
    const int rr = (int)ceilf(3.f * sqrtf(lam));
    const float itz = 1.f / tz;
    const float u = cam.fx * G.tx * itz + cam.cx;
    const float v = cam.fy * G.ty * itz + cam.cy;
    const float fr = (float)rr;
    const int x0 = (int)fminf(fmaxf(floorf((u - fr) * (1.f / kTile)), 0.f), (float)cam.tiles_x);
    const int y0 = (int)fminf(fmaxf(floorf((v - fr) * (1.f / kTile)), 0.f), (float)cam.tiles_y);
    const int x1 = (int)fminf(fmaxf(floorf((u + fr) * (1.f / kTile)) + 1.f, 0.f), (float)cam.tiles_x);
    const int y1 = (int)fminf(fmaxf(floorf((v + fr) * (1.f / kTile)) + 1.f, 0.f), (float)cam.tiles_y);
    if (x0 < x1 && y0 < y1) {
      r = rr;
      touched = (unsigned)((x1 - x0) * (y1 - y0));
      uvo = make_float2(u, v);
      const float o = 1.f / (1.f + expf(-p.logits[i]));
      co = make_float4(G.c * idet, -G.b * idet, G.a * idet, o);
      // colour at the view direction from the camera centre
      const float dx = p.means[3 * i] - cam.campos[0];
      const float dy = p.means[3 * i + 1] - cam.campos[1];
      const float dz = p.means[3 * i + 2] - cam.campos[2];
      const float il = 1.f / sqrtf(dx * dx + dy * dy + dz * dz);
      float Y[16];
      sh_eval(K, DEG, dx * il, dy * il, dz * il, Y, nullptr);
      const float* sh = buf + lane * P;
#pragma unroll
      for (int ch = 0; ch < 3; ++ch) {
        float acc = 0.5f;
#pragma unroll
        for (int k = 0; k < D; ++k) acc += Y[k] * sh[3 * k + ch];
        col[ch] = fmaxf(acc, 0.f);
      }
    }
  }
  radius[i] = r;
  tiles_touched[i] = touched;
  uv[i] = uvo;
  conic_op[i] = co;
  rgb[3 * i] = col[0];
  rgb[3 * i + 1] = col[1];
  rgb[3 * i + 2] = col[2];
}

struct Grads {
  float* means;
  float* log_scales;
  float* quats;
  float* logits;
  float* sh;
};

template <int DEG>
__device__ __forceinline__ void project_bwd_one(const Params& p, int n, int i, const Cam& cam,
                                                const Opts& op, const SHConst& K,
                                                const float* grad2d, const Grads& out,
                                                float* shrow) {
  constexpr int D = ShLayout<DEG>::D;
  if (i >= n) return;
  const float* g9 = grad2d + 9 * (size_t)i;
  float gin[9];
  bool any = false;
#pragma unroll
  for (int k = 0; k < 9; ++k) { gin[k] = g9[k]; any |= gin[k] != 0.f; }
  const float mx = p.means[3 * i], my = p.means[3 * i + 1], mz = p.means[3 * i + 2];
  const float tz = view_depth(cam, mx, my, mz);
  if (!any || !(tz > op.near_z)) {   // no contribution: every gradient is 0
    for (int k = 0; k < 3; ++k) { out.means[3 * i + k] = 0.f; out.log_scales[3 * i + k] = 0.f; }
    for (int k = 0; k < 4; ++k) out.quats[4 * i + k] = 0.f;
    out.logits[i] = 0.f;
#pragma unroll
    for (int k = 0; k < 3 * D; ++k) shrow[k] = 0.f;
    return;
  }
  Geo G;
  geometry(cam, op, p, i, tz, G);
  const float gu = gin[0], gv = gin[1], gQa = gin[2], gQb = gin[3], gQc = gin[4], go = gin[5];
  float gmu[3] = {0.f, 0.f, 0.f};
  // ---- opacity = sigmoid(logit)
  const float o = 1.f / (1.f + expf(-p.logits[i]));
  out.logits[i] = go * o * (1.f - o);
  // ---- colour: rgb = max(0, sum_k Y_k(dir) sh_k + 0.5), dir = (mu - campos)/|mu - campos|
  {
    const float dx = mx - cam.campos[0], dy = my - cam.campos[1], dz = mz - cam.campos[2];
    const float il = 1.f / sqrtf(dx * dx + dy * dy + dz * dz);
    const float d[3] = {dx * il, dy * il, dz * il};
    float Y[16], dY[16][3];
    sh_eval(K, DEG, d[0], d[1], d[2], Y, dY);
    float gdir[3] = {0.f, 0.f, 0.f};
#pragma unroll
    for (int ch = 0; ch < 3; ++ch) {
      float raw = 0.5f;
#pragma unroll
      for (int k = 0; k < D; ++k) raw += Y[k] * shrow[3 * k + ch];
      const float gc = raw < 0.f ? 0.f : gin[6 + ch];
#pragma unroll
      for (int k = 0; k < D; ++k) {
        const float s = shrow[3 * k + ch] * gc;
        shrow[3 * k + ch] = Y[k] * gc;             // the coefficient's gradient, in place
        gdir[0] += s * dY[k][0]; gdir[1] += s * dY[k][1]; gdir[2] += s * dY[k][2];
      }
    }
    const float dd = d[0] * gdir[0] + d[1] * gdir[1] + d[2] * gdir[2];
    for (int k = 0; k < 3; ++k) gmu[k] += (gdir[k] - d[k] * dd) * il;
  }
  // ---- conic = (c, -b, a)/det  ->  (a, b, c) of the dilated 2-D covariance
  const float a = G.a, b = G.b, c = G.c, det = G.det;
  const float id2 = 1.f / (det * det);
  const float ga = (-gQa * c * c + gQb * b * c - gQc * b * b) * id2;
  const float gb = (2.f * gQa * b * c - gQb * (det + 2.f * b * b) + 2.f * gQc * a * b) * id2;
  const float gc = (-gQa * b * b + gQb * a * b - gQc * a * a) * id2;
  // ---- a = |P0|^2 + dil, b = P0.P1, c = |P1|^2 + dil
  float gP[2][3];
  for (int k = 0; k < 3; ++k) {
    gP[0][k] = 2.f * ga * G.P[0][k] + gb * G.P[1][k];
    gP[1][k] = gb * G.P[0][k] + 2.f * gc * G.P[1][k];
  }
  // ---- P = T M
  float gT[2][3], gM[3][3];
  for (int r = 0; r < 2; ++r)
    for (int j = 0; j < 3; ++j)
      gT[r][j] = gP[r][0] * G.M[j][0] + gP[r][1] * G.M[j][1] + gP[r][2] * G.M[j][2];
  for (int j = 0; j < 3; ++j)
    for (int k = 0; k < 3; ++k) gM[j][k] = gP[0][k] * G.T[0][j] + gP[1][k] * G.T[1][j];
  // ---- M = R(q) diag(s), s = exp(log_scale)
  float gR[3][3];
  for (int k = 0; k < 3; ++k) {
    float gs = 0.f;
    for (int j = 0; j < 3; ++j) { gR[j][k] = gM[j][k] * G.s[k]; gs += gM[j][k] * G.Rq[j][k]; }
    out.log_scales[3 * i + k] = gs * G.s[k];
  }
  // ---- R(q) of the unit quaternion (w, x, y, z), then the normalisation q/|q|
  {
    const float w = G.qw, x = G.qx, y = G.qy, z = G.qz;
    const float gw = 2.f * (-z * gR[0][1] + y * gR[0][2] + z * gR[1][0] - x * gR[1][2] - y * gR[2][0] + x * gR[2][1]);
    const float gx = 2.f * (y * gR[0][1] + z * gR[0][2] + y * gR[1][0] - 2.f * x * gR[1][1] - w * gR[1][2] +
                            z * gR[2][0] + w * gR[2][1] - 2.f * x * gR[2][2]);
    const float gy = 2.f * (-2.f * y * gR[0][0] + x * gR[0][1] + w * gR[0][2] + x * gR[1][0] + z * gR[1][2] -
                            w * gR[2][0] + z * gR[2][1] - 2.f * y * gR[2][2]);
    const float gz = 2.f * (-2.f * z * gR[0][0] - w * gR[0][1] + x * gR[0][2] + w * gR[1][0] - 2.f * z * gR[1][1] +
                            y * gR[1][2] + x * gR[2][0] + y * gR[2][1]);
    const float dot = w * gw + x * gx + y * gy + z * gz;
    out.quats[4 * i + 0] = (gw - w * dot) * G.qinv;
    out.quats[4 * i + 1] = (gx - x * dot) * G.qinv;
    out.quats[4 * i + 2] = (gy - y * dot) * G.qinv;
    out.quats[4 * i + 3] = (gz - z * dot) * G.qinv;
  }
  // ---- T = J W
  float gJ00 = 0.f, gJ02 = 0.f, gJ11 = 0.f, gJ12 = 0.f;
  for (int k = 0; k < 3; ++k) {
    gJ00 += gT[0][k] * cam.R[k];
    gJ02 += gT[0][k] * cam.R[6 + k];
    gJ11 += gT[1][k] * cam.R[3 + k];
    gJ12 += gT[1][k] * cam.R[6 + k];
  }
  // ---- J(t) with the guarded x' = clamp(x/z) z  (true derivative on both sides)
  const float itz = 1.f / tz, itz2 = itz * itz, itz3 = itz2 * itz;
  float gtx = 0.f, gty = 0.f;
  float gtz = -cam.fx * itz2 * gJ00 - cam.fy * itz2 * gJ11;
  if (!G.clx) { gtx += -cam.fx * itz2 * gJ02; gtz += 2.f * cam.fx * G.tx * itz3 * gJ02; }
  else { const float L = G.tx > 0.f ? cam.limx : -cam.limx; gtz += cam.fx * L * itz2 * gJ02; }
  if (!G.cly) { gty += -cam.fy * itz2 * gJ12; gtz += 2.f * cam.fy * G.ty * itz3 * gJ12; }
  else { const float L = G.ty > 0.f ? cam.limy : -cam.limy; gtz += cam.fy * L * itz2 * gJ12; }
  // ---- uv = (fx tx/tz + cx, fy ty/tz + cy)
  gtx += gu * cam.fx * itz;
  gty += gv * cam.fy * itz;
  gtz += -(gu * cam.fx * G.tx + gv * cam.fy * G.ty) * itz2;
  // ---- t = W mu + t_cam
  for (int k = 0; k < 3; ++k)
    out.means[3 * i + k] = gmu[k] + cam.R[k] * gtx + cam.R[3 + k] * gty + cam.R[6 + k] * gtz;
}

template <int DEG>
__global__ void __launch_bounds__(kProjThreads)
project_bwd_kernel(Params p, int n, Cam cam, Opts op, SHConst K, const float* grad2d,
                   Grads out) {
  pdl_prologue();
  constexpr int P = ShLayout<DEG>::P;
  __shared__ float s_sh[kProjThreads / 32][32 * P];
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31, first = i - lane;
  if (first >= n) return;                                  // whole warp
  float* buf = s_sh[threadIdx.x >> 5];
  sh_to_shared<DEG>(p.sh, n, first, buf);
  // every lane's sh row is replaced by its gradient in place, then written out together
  project_bwd_one<DEG>(p, n, i, cam, op, K, grad2d, out, buf + lane * P);
  sh_from_shared<DEG>(out.sh, n, first, buf);
}

Params params_of(const abcd_gaussians* g) {
  return Params{g->means, g->log_scales, g->quats, g->opacity_logits, g->sh};
}

bool gaussians_ok(const abcd_gaussians* g) {
  return g && g->n >= 0 && g->sh_degree >= 0 && g->sh_degree <= 3 &&
         (g->n == 0 || (g->means && g->log_scales && g->quats && g->opacity_logits && g->sh)) &&
         ((uintptr_t)g->quats & 15) == 0;
}

bool camera_ok(const abcd_camera* c) {
  return c && c->width > 0 && c->height > 0 && c->fx > 0.f && c->fy > 0.f &&
         (long long)((c->width + kTile - 1) / kTile) * ((c->height + kTile - 1) / kTile) < (1LL << 24);
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_project(abcd_ctx* ctx, const abcd_gaussians* theta,
                                    const abcd_camera* cam, const abcd_render_opts* opts,
                                    abcd_projected* out) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!gaussians_ok(theta)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project: bad gaussians (null pointer, degree or unaligned quats)");
  if (!camera_ok(cam)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project: bad camera");
  if (!out || (theta->n > 0 && (!out->uv || !out->conic_opacity || !out->rgb || !out->depth ||
                                !out->radius || !out->tiles_touched)))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project: null output");
  if (((uintptr_t)out->uv & 7) || ((uintptr_t)out->conic_opacity & 15))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project: uv must be 8-byte and conic_opacity 16-byte aligned");
  if (theta->n == 0) return ABCD_OK;
  const int blocks = (theta->n + kProjThreads - 1) / kProjThreads;
  void (*kern)(Params, int, Cam, Opts, SHConst, float2*, float4*, float*, float*, int*, unsigned*) =
      theta->sh_degree == 0 ? project_fwd_kernel<0> : theta->sh_degree == 1 ? project_fwd_kernel<1>
      : theta->sh_degree == 2 ? project_fwd_kernel<2> : project_fwd_kernel<3>;
  return check_launch(ctx, "project_fwd_kernel",
                      launch_pdl(kern, dim3(blocks), dim3(kProjThreads), 0, ctx->stream,
                                 params_of(theta), theta->n, make_cam(cam, opts), make_opts(opts),
                                 ctx->sh, (float2*)out->uv, (float4*)out->conic_opacity, out->rgb,
                                 out->depth, out->radius, out->tiles_touched));
}

extern "C" abcd_status abcd_project_backward(abcd_ctx* ctx, const abcd_gaussians* theta,
                                             const abcd_camera* cam, const abcd_render_opts* opts,
                                             const float* grad2d, abcd_gaussians* grads) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!gaussians_ok(theta) || !gaussians_ok(grads) || grads->n != theta->n ||
      grads->sh_degree != theta->sh_degree)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project_backward: bad gaussians/grads");
  if (!camera_ok(cam)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project_backward: bad camera");
  if (theta->n > 0 && !grad2d) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_project_backward: null grad2d");
  if (theta->n == 0) return ABCD_OK;
  const int blocks = (theta->n + kProjThreads - 1) / kProjThreads;
  void (*kern)(Params, int, Cam, Opts, SHConst, const float*, Grads) =
      theta->sh_degree == 0 ? project_bwd_kernel<0> : theta->sh_degree == 1 ? project_bwd_kernel<1>
      : theta->sh_degree == 2 ? project_bwd_kernel<2> : project_bwd_kernel<3>;
  return check_launch(ctx, "project_bwd_kernel",
                      launch_pdl(kern, dim3(blocks), dim3(kProjThreads), 0, ctx->stream,
                                 params_of(theta), theta->n, make_cam(cam, opts), make_opts(opts),
                                 ctx->sh, grad2d,
                                 Grads{grads->means, grads->log_scales, grads->quats,
                                       grads->opacity_logits, grads->sh}));
}
