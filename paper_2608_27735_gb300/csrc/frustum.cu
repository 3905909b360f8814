// a0: which camera-partition pairs are visible (Section 2 stores renders for the visible
// camera-partition pairs and trains a block on the cameras that observe its partition; the
// paper's runtime discussion speaks of the pairs left "after frustum filtering").
//
// A partition's extent is the axis-aligned box of its cell and of every one of its Gaussians'
// 3-sigma ellipsoids: for covariance Sigma = R(q) diag(s^2) R(q)^T the ellipsoid
// {x : (x - mu)^T Sigma^-1 (x - mu) <= 9} reaches mu_k +- 3 sqrt(Sigma_kk) along axis k.
// abcd_block_bounds computes the Gaussians' box on the device (one CTA: a per-stage operation,
// not a per-step one).  abcd_pair_visible tests a box against the camera's view frustum in
// camera space, {z >= near_z, |x| <= gx z, |y| <= gy z} with gx, gy the guard-widened half
// fields of view: the pair is culled only when the whole box lies outside one of those five
// half-spaces, so no pair whose box meets the frustum is ever culled.
#include <cmath>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

constexpr int kBoundsThreads = 1024;

__global__ void __launch_bounds__(kBoundsThreads)
bounds_kernel(const float* __restrict__ means, const float* __restrict__ log_scales,
              const float* __restrict__ quats, int n, float* box) {
  pdl_prologue();
  float lo[3] = {INFINITY, INFINITY, INFINITY}, hi[3] = {-INFINITY, -INFINITY, -INFINITY};
  for (int i = threadIdx.x; i < n; i += kBoundsThreads) {
    float q[4];
    for (int k = 0; k < 4; ++k) q[k] = quats[4 * i + k];
    const float qn = rsqrtf(fmaxf(q[0] * q[0] + q[1] * q[1] + q[2] * q[2] + q[3] * q[3], 1e-30f));
    const float w = q[0] * qn, x = q[1] * qn, y = q[2] * qn, z = q[3] * qn;
    // rotation matrix of the unit quaternion (w, x, y, z), rows r0..r2
    const float R[9] = {1.f - 2.f * (y * y + z * z), 2.f * (x * y - w * z), 2.f * (x * z + w * y),
                        2.f * (x * y + w * z), 1.f - 2.f * (x * x + z * z), 2.f * (y * z - w * x),
                        2.f * (x * z - w * y), 2.f * (y * z + w * x), 1.f - 2.f * (x * x + y * y)};
    float s[3];
    for (int j = 0; j < 3; ++j) s[j] = expf(log_scales[3 * i + j]);
    for (int k = 0; k < 3; ++k) {
      float var = 0.f;
      for (int j = 0; j < 3; ++j) { const float a = R[3 * k + j] * s[j]; var = fmaf(a, a, var); }
      // 1e-6 relative widening: the box holds the ellipsoid whatever the fp32 rounding above
      const float ext = 3.f * sqrtf(var) * (1.f + 1e-6f) + 1e-7f;
      const float m = means[3 * i + k];
      lo[k] = fminf(lo[k], m - ext);
      hi[k] = fmaxf(hi[k], m + ext);
    }
  }
  __shared__ float red[6][kBoundsThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int k = 0; k < 3; ++k) {
    float a = lo[k], b = hi[k];
    for (int o = 16; o > 0; o >>= 1) {
      a = fminf(a, __shfl_xor_sync(0xffffffffu, a, o));
      b = fmaxf(b, __shfl_xor_sync(0xffffffffu, b, o));
    }
    if (lane == 0) { red[k][wid] = a; red[3 + k][wid] = b; }
  }
  __syncthreads();
  if (threadIdx.x < 6) {
    float v = red[threadIdx.x][0];
    for (int j = 1; j < kBoundsThreads / 32; ++j)
      v = threadIdx.x < 3 ? fminf(v, red[threadIdx.x][j]) : fmaxf(v, red[threadIdx.x][j]);
    box[threadIdx.x] = v;
  }
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_block_bounds(abcd_ctx* ctx, const abcd_gaussians* theta, float* box) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!theta || theta->n < 0 || !box || (theta->n > 0 && (!theta->means || !theta->log_scales || !theta->quats)))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_block_bounds: bad arguments");
  return check_launch(ctx, "bounds_kernel",
                      launch_pdl(bounds_kernel, dim3(1), dim3(kBoundsThreads), 0, ctx->stream,
                                 (const float*)theta->means, (const float*)theta->log_scales,
                                 (const float*)theta->quats, theta->n, box));
}

extern "C" abcd_status abcd_pair_visible(const abcd_camera* cam, const abcd_render_opts* opts,
                                         const double box[6], int* visible) {
  if (!cam || !box || !visible || cam->width <= 0 || cam->height <= 0 || !(cam->fx > 0) ||
      !(cam->fy > 0))
    return ABCD_ERR_INVALID_ARG;
  if (!(box[0] <= box[3] && box[1] <= box[4] && box[2] <= box[5])) {   // empty (or NaN) box
    *visible = 0;
    return ABCD_OK;
  }
  const Opts op = make_opts(opts);
  const double gx = (double)op.guard * 0.5 * cam->width / cam->fx;
  const double gy = (double)op.guard * 0.5 * cam->height / cam->fy;
  // the five half-spaces n . p_cam + d >= 0 of the frustum in camera space
  const double pl[5][4] = {{0, 0, 1, -(double)op.near_z},
                           {-1, 0, gx, 0}, {1, 0, gx, 0},
                           {0, -1, gy, 0}, {0, 1, gy, 0}};
  int vis = 1;
  for (int p = 0; p < 5 && vis; ++p) {
    // in world space: (R^T n) . x + (n . t + d); its largest value over the box
    double a[3], c = pl[p][3];
    for (int j = 0; j < 3; ++j) {
      a[j] = 0.0;
      for (int i = 0; i < 3; ++i) a[j] += pl[p][i] * (double)cam->R[3 * i + j];
    }
    for (int i = 0; i < 3; ++i) c += pl[p][i] * (double)cam->t[i];
    double best = c;
    for (int j = 0; j < 3; ++j) best += a[j] > 0 ? a[j] * box[3 + j] : a[j] * box[j];
    if (best < 0.0) vis = 0;
  }
  *visible = vis;
  return ABCD_OK;
}
