// abcd_backward: the backward pass of one active-block step (Section 2: the step's loss is
// differentiated with respect to the active block's parameters and nothing else):
// K6 loss (optional) -> K7 blend/composite backward -> K8 projection backward.
#include "abcd_internal.cuh"

using namespace abcd;

extern "C" abcd_status abcd_backward(abcd_ctx* ctx, const abcd_gaussians* theta,
                                     const abcd_camera* cam, const abcd_render_opts* opts,
                                     const abcd_projected* proj, const abcd_tiles* tiles,
                                     const void* F, const void* B, int fb_dtype, const float* bg,
                                     const float* out_rgba, const abcd_fwd_state* state,
                                     const float* gt_rgb, float lambda_ssim, float* loss_out,
                                     const float* dL_dout, abcd_gaussians* grads) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_backward: no workspace");
  if (!theta || !cam) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_backward: null theta or camera");
  if (theta->n > ctx->max_g) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_backward: n exceeds workspace");
  const long long npix = (long long)cam->width * cam->height;
  const float* g = dL_dout;
  abcd_status s;
  if (gt_rgb) {
    if (npix > ctx->max_pixels) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_backward: image exceeds workspace");
    if ((s = loss_launch(ctx, out_rgba, gt_rgb, cam->width, cam->height, lambda_ssim, loss_out,
                         ctx->ws.dl_dout)))
      return s;
    g = ctx->ws.dl_dout;
  } else if (!g) {
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_backward: need gt_rgb or dL_dout");
  }
  if ((s = abcd_render_backward(ctx, cam, opts, proj, tiles, F, B, fb_dtype, bg, state, g,
                                theta->n, ctx->ws.grad2d)))
    return s;
  return abcd_project_backward(ctx, theta, cam, opts, ctx->ws.grad2d, grads);
}

extern "C" abcd_status abcd_train_step(abcd_ctx* ctx, abcd_gaussians* theta, abcd_gaussians* grads,
                                       abcd_gaussians* m, abcd_gaussians* v,
                                       const abcd_camera* cam, const abcd_render_opts* opts,
                                       abcd_projected* proj, abcd_tiles* tiles, const void* F,
                                       const void* B, int fb_dtype, const float* bg,
                                       float* out_rgba, abcd_fwd_state* state,
                                       const float* gt_rgb, float lambda_ssim, float* loss_out,
                                       const float lr[6], float beta1, float beta2, float eps,
                                       int step) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!theta || !grads || !m || !v || !cam || !proj || !tiles || !out_rgba || !state || !gt_rgb || !lr)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_train_step: null argument");
  abcd_status s;
  if ((s = abcd_project(ctx, theta, cam, opts, proj))) return s;
  if ((s = abcd_bin_sort(ctx, proj, theta->n, cam, opts, tiles))) return s;
  if ((s = abcd_render_composite_fwd(ctx, cam, opts, proj, tiles, F, B, fb_dtype, bg, out_rgba,
                                     state, nullptr)))
    return s;
  if ((s = abcd_backward(ctx, theta, cam, opts, proj, tiles, F, B, fb_dtype, bg, out_rgba, state,
                         gt_rgb, lambda_ssim, loss_out, nullptr, grads)))
    return s;
  return abcd_adam_active(ctx, theta, grads, m, v, lr, beta1, beta2, eps, step);
}

extern "C" abcd_status abcd_refresh_layer(abcd_ctx* ctx, const abcd_gaussians* theta,
                                          const abcd_camera* cam, const abcd_render_opts* opts,
                                          abcd_projected* proj, abcd_tiles* tiles, int* tile_map,
                                          void* packed, int* count) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!theta || !cam || !proj || !tiles)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_refresh_layer: null argument");
  abcd_status s;
  if ((s = abcd_project(ctx, theta, cam, opts, proj))) return s;
  if ((s = abcd_bin_sort(ctx, proj, theta->n, cam, opts, tiles))) return s;
  return abcd_render_refresh_packed(ctx, cam, opts, proj, tiles, tile_map, packed, count);
}
