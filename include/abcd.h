/* libabcd -- GB300 (sm_103a) hot path of ABCD, Alpha-Composited Block Coordinate Descent.
 *
 * ABCD trains one spatial block of 3D Gaussians at a time (Section 2).  The frozen blocks
 * that lie in front of / behind the active partition, seen from a camera, are collapsed by
 * associativity of alpha compositing into two premultiplied RGBA images F and B; every
 * training step renders only the active block A and composites F over A over B, evaluates
 * the reconstruction loss and backpropagates into the active block only.  The renderer is
 * 3D Gaussian Splatting (Section 1, last paragraph).
 *
 * Conventions for every call:
 *  - Tensor arguments are DEVICE pointers owned by the caller, fp32 unless stated, C order.
 *  - Struct arguments (camera, options, pointer bundles) are HOST structs read during the
 *    call; nothing keeps a reference to them after it returns.
 *  - Every compute call is asynchronous on the context's CUDA stream and returns a status.
 *    Argument errors are reported before anything is launched (ABCD_ERR_INVALID_ARG).
 *    Errors found on the device (tile-list capacity, bounds) are OR-ed into a device status
 *    word that abcd_sync() reads.  No call allocates device memory, synchronizes the
 *    device, throws, traps or exits; scratch comes from the caller's workspace.
 *  - The library never touches parameters outside the active block it is given.
 */
#ifndef ABCD_H
#define ABCD_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ABCD_OK = 0,
  ABCD_ERR_INVALID_ARG = 1,   /* bad pointer / size / option; nothing launched */
  ABCD_ERR_CUDA = 2,          /* a CUDA runtime call or launch failed (see abcd_last_error) */
  ABCD_ERR_CAPACITY = 3,      /* device: tile pairs K exceeded abcd_tiles.capacity */
  ABCD_ERR_TIMEOUT = 4,       /* device: a bounded wait gave up (the radix sort's look-back;
                                 the results of that call are wrong, nothing hangs) */
  ABCD_ERR_WORKSPACE = 5      /* workspace missing or smaller than abcd_workspace_size() */
} abcd_status;

typedef struct abcd_ctx abcd_ctx;

/* Pinhole camera: x_cam = R * x_world + t (R row-major), x right, y down, z forward;
 * pixel (i, j) covers [i, i+1) x [j, j+1), so its centre is (i + 0.5, j + 0.5) and a camera
 * point projects to (fx x/z + cx, fy y/z + cy). */
typedef struct {
  float R[9];
  float t[3];
  float fx, fy, cx, cy;
  int width, height;
} abcd_camera;

/* Renderer constants of 3D Gaussian Splatting.  Pass NULL for the defaults in brackets. */
typedef struct {
  float near_z;     /* cull Gaussians with camera depth <= near_z [0.2] */
  float dilation;   /* added to the diagonal of the 2-D covariance [0.3] */
  float guard;      /* Jacobian uses x/z, y/z clamped to guard * tan(fov/2) [1.3] */
  float alpha_max;  /* alpha = min(alpha_max, o exp(-sigma)) [0.99] */
  float alpha_min;  /* contributions with alpha < alpha_min are skipped [1/255] */
  float t_min;      /* a pixel stops before a Gaussian that would take T below t_min [1e-4] */
} abcd_render_opts;

/* Parameters of the active block (SoA, device).  Shapes: means [n][3], log_scales [n][3],
 * quats [n][4] as (w, x, y, z), not necessarily unit, opacity_logits [n],
 * sh [n][D][3] with D = (sh_degree + 1)^2 and coefficient index l*l + l + m (real SH,
 * Condon-Shortley phase).  The same struct carries gradients and Adam moments. */
typedef struct {
  float* means;
  float* log_scales;
  float* quats;
  float* opacity_logits;
  float* sh;
  int n;
  int sh_degree;    /* 0..3 */
} abcd_gaussians;

/* Output of abcd_project (device, length n each).  A Gaussian is visible iff radius > 0. */
typedef struct {
  float* uv;             /* [n][2] pixel-space mean */
  float* conic_opacity;  /* [n][4] (a, b, c, opacity): inverse 2-D covariance [[a,b],[b,c]] */
  float* rgb;            /* [n][3] view-dependent colour, clamped at 0 */
  float* depth;          /* [n] camera-space depth (sort key) */
  int* radius;           /* [n] ceil(3 sqrt(lambda_max)) in pixels, 0 = culled */
  unsigned* tiles_touched; /* [n] 16x16 tiles met by the square of half-side radius */
} abcd_projected;

/* Per-tile Gaussian lists (device).  For tile t = ty * tiles_x + tx (16x16 tiles,
 * tiles_x = ceil(W/16)), ids[ranges[2t] .. ranges[2t+1]) are the Gaussians listed on the tile
 * (see abcd_bin_sort), front to back by (fp32 depth, id). */
typedef struct {
  unsigned* ids;         /* [capacity] */
  unsigned* ranges;      /* [tiles_x * tiles_y][2] */
  long long capacity;    /* entries available in ids (<= the workspace's max_pairs) */
  long long* count;      /* device scalar: K, the number of (tile, Gaussian) pairs.  If
                            K > capacity, ABCD_ERR_CAPACITY is raised, ranges are all empty
                            and *count still holds the required K. */
} abcd_tiles;

/* Per-pixel state saved by the forward pass for the backward pass (device). */
typedef struct {
  float* A_T;            /* [H][W][4]: active premultiplied rgb and its final transmittance */
  unsigned* n_last;      /* [H][W]: list positions walked up to the last contributor */
} abcd_fwd_state;

enum { ABCD_F16 = 0, ABCD_F32 = 1 };   /* element type of F, B and cached layers */

/* ---- context, stream, workspace ------------------------------------------------------ */
abcd_status abcd_create(abcd_ctx** ctx, int device, void* cuda_stream);
abcd_status abcd_destroy(abcd_ctx* ctx);
abcd_status abcd_set_stream(abcd_ctx* ctx, void* cuda_stream);
/* Bytes of device scratch for blocks of up to max_gaussians, up to max_pairs tile pairs
 * and images of up to max_pixels pixels. */
abcd_status abcd_workspace_size(int max_gaussians, long long max_pairs, long long max_pixels,
                                size_t* bytes);
/* Hands the context a caller-owned device buffer (>= abcd_workspace_size bytes, 256-byte
 * aligned).  Clears the device status word (asynchronously, on the context's stream). */
abcd_status abcd_set_workspace(abcd_ctx* ctx, void* device_ptr, size_t bytes,
                               int max_gaussians, long long max_pairs, long long max_pixels);
/* Waits for the stream, then returns the first device-detected error (sticky) or ABCD_OK. */
abcd_status abcd_sync(abcd_ctx* ctx);
abcd_status abcd_clear_status(abcd_ctx* ctx);
const char* abcd_last_error(const abcd_ctx* ctx);
/* Number of kernels this context has launched since creation (instrumentation). */
long long abcd_launch_count(const abcd_ctx* ctx);
/* Bound on the polls of a device-side wait (the radix sort's decoupled look-back waits for the
 * tiles before its own, whose CTAs are already running) [2^20, about 40 ms]: a wait that
 * reaches it gives up, the call's results are wrong and ABCD_ERR_TIMEOUT is set in the status
 * word (abcd_sync); nothing hangs, and later calls run normally once the status is cleared. */
abcd_status abcd_set_wait_limit(abcd_ctx* ctx, unsigned polls);
/* Test hook for the bounded waits: in the next abcd_bin_sort call, look-back tile `tile` (2048
 * keys) of the first pass of the depth sort publishes nothing, so the waits of the tiles after
 * it run out (after the wait limit).  -1 (the default) turns it off; it turns itself off after
 * that pass. */
abcd_status abcd_test_withhold_lookback(abcd_ctx* ctx, long long tile);

/* ---- the hot path (Section 2: one step renders only the active block) ----------------- */

/* K2. EWA projection of the active block for one camera.  Section 2 renders only the active
 * partition at each step; the renderer is 3D Gaussian Splatting, which the paper instantiates
 * by citation (Section 1, last paragraph), so the formulas are 3DGS's: camera-space mean, world
 * covariance R(q) diag(exp(2 log_scale)) R(q)^T, 2-D covariance J W Sigma W^T J^T +
 * dilation*I, its inverse, the 3-sigma radius, SH colour + 0.5 clamped at 0 and
 * opacity = sigmoid(logit).  Writes every field of out. */
abcd_status abcd_project(abcd_ctx* ctx, const abcd_gaussians* theta, const abcd_camera* cam,
                         const abcd_render_opts* opts, abcd_projected* out);

/* K3 + K4. Tile binning and depth sort of the active block (the tile rasteriser of 3D Gaussian
 * Splatting, Section 1 by citation; Section 2 renders the active partition alone, so only its
 * Gaussians are binned).  A visible Gaussian is listed in each tile its square
 * [u-r, u+r] x [v-r, v+r] meets on which it comes within a small margin of alpha_min: the least
 * sigma over the box of the tile's pixel centres, in log2 units, is at most
 * (1.001 log2(opacity / alpha_min) + 0.01) 1.001 (the exact rule, sigma <= ln(opacity /
 * alpha_min), widened so that fp32 rounding never drops a tile it keeps; a list may hold a few
 * entries that every pixel of the tile skips); lists are ordered by the fp32 depth, ties by id.  Leaving out the tiles on which
 * every pixel would skip the Gaussian does not change any pixel.  n must equal the n given
 * to abcd_project; opts as there (NULL = defaults; alpha_min is used).  Also leaves in the
 * context's workspace the tiles ordered by decreasing list length, tagged with out->ranges;
 * the render calls given these same ranges launch their longest tiles first (a scheduling
 * hint only: no result depends on it). */
abcd_status abcd_bin_sort(abcd_ctx* ctx, const abcd_projected* proj, int n,
                          const abcd_camera* cam, const abcd_render_opts* opts, abcd_tiles* out);

/* K5. The active partition rendered and composited with the cached foreground and background
 * (Section 2: the frozen partitions in front of / behind the active one collapse into F and B,
 * and compositing with them equals rendering with every frozen parameter present).  The call
 * takes the active block's projection (abcd_project) and tile lists (abcd_bin_sort) rather than
 * theta itself, so that one projection serves the forward, the backward and the refresh.
 * Front-to-back blend of the active block per pixel (alpha = min(alpha_max,
 * o exp(-sigma)), skip alpha < alpha_min, stop before T < t_min), giving the premultiplied
 * A = (sum T_i alpha_i c_i, 1 - T_final); then out = F over (A over B), over meaning
 * X + (1 - X.a) Y on premultiplied RGBA, and out.rgb += (1 - out.a) * bg.
 * F, B: [H][W][4] of fb_dtype, or NULL for transparent.  bg: 3 host floats or NULL (0).
 * out_rgba: [H][W][4] fp32 (may be NULL).  state: may be NULL (no backward).
 * refresh_f16: optional [H][W][4] fp16 receiving A alone (the cache refresh of Section 2). */
abcd_status abcd_render_composite_fwd(abcd_ctx* ctx, const abcd_camera* cam,
                                      const abcd_render_opts* opts, const abcd_projected* proj,
                                      const abcd_tiles* tiles, const void* F, const void* B,
                                      int fb_dtype, const float* bg, float* out_rgba,
                                      abcd_fwd_state* state, void* refresh_f16);

/* K6. The reconstruction loss each step of Section 2 evaluates, in the L1 + D-SSIM form of
 * 3D Gaussian Splatting: (1 - lambda) mean|x - y| + lambda (1 - mean SSIM(x, y)) over the
 * rgb of out_rgba [H][W][4] against gt_rgb [H][W][3]; SSIM with an 11x11 Gaussian window
 * (sigma 1.5), zero padding, C1 = 0.01^2, C2 = 0.03^2.  loss_out: device float scalar (may
 * be NULL).  dL_dout: [H][W][3] receives dL/d(out.rgb) (may be NULL: the loss alone).  The
 * SSIM's per-pixel partials pass between its two kernels through the workspace, so the image
 * may have at most the workspace's max_pixels pixels (ABCD_ERR_WORKSPACE otherwise, before any
 * launch); ABCD_ERR_INVALID_ARG for null inputs, non-positive sizes or lambda outside [0, 1]. */
abcd_status abcd_loss(abcd_ctx* ctx, const float* out_rgba, const float* gt_rgb, int width,
                      int height, float lambda_ssim, float* loss_out, float* dL_dout);

/* K7. Backward of the blend + composite for one image (Section 2: gradients flow only into the
 * active block; F and B are constants of the step): given dL/d(final rgb) [H][W][3],
 * writes grad2d [n][9] = dL/d(u, v, a, b, c, opacity, r, g, b) per Gaussian (overwritten).
 * The alpha of the active layer also receives -(1 - F.a) <g, B.rgb + (1 - B.a) bg>. */
abcd_status abcd_render_backward(abcd_ctx* ctx, const abcd_camera* cam,
                                 const abcd_render_opts* opts, const abcd_projected* proj,
                                 const abcd_tiles* tiles, const void* F, const void* B,
                                 int fb_dtype, const float* bg, const abcd_fwd_state* state,
                                 const float* dL_dout, int n, float* grad2d);

/* K8. Chain rule from grad2d [n][9] to the parameters of theta, the active block (Section 2:
 * gradients reach theta_active only; the projection is 3DGS's, Section 1 by citation).
 * Overwrites grads; culled Gaussians get 0. */
abcd_status abcd_project_backward(abcd_ctx* ctx, const abcd_gaussians* theta,
                                  const abcd_camera* cam, const abcd_render_opts* opts,
                                  const float* grad2d, abcd_gaussians* grads);

/* K6 + K7 + K8: the backward pass of one step into the active block only.  With gt_rgb,
 * evaluates the loss into loss_out and uses its gradient; with gt_rgb == NULL, dL_dout is
 * the given upstream gradient.  grad2d and dL/dout live in the workspace. */
abcd_status abcd_backward(abcd_ctx* ctx, const abcd_gaussians* theta, const abcd_camera* cam,
                          const abcd_render_opts* opts, const abcd_projected* proj,
                          const abcd_tiles* tiles, const void* F, const void* B, int fb_dtype,
                          const float* bg, const float* out_rgba, const abcd_fwd_state* state,
                          const float* gt_rgb, float lambda_ssim, float* loss_out,
                          const float* dL_dout, abcd_gaussians* grads);

/* K9. The update of the T gradient steps of Section 2 on theta_active (the optimiser is Adam, as
 * in 3D Gaussian Splatting; the paper names none).  Bias-corrected (torch semantics), dense
 * over the active block only:
 * m = b1 m + (1-b1) g; v = b2 v + (1-b2) g^2; theta -= lr m/(1-b1^t) / (sqrt(v/(1-b2^t)) + eps).
 * lr[6] per group: means, log_scales, quats, opacity_logits, sh degree 0, sh degree >= 1.
 * step is 1-based. */
abcd_status abcd_adam_active(abcd_ctx* ctx, abcd_gaussians* theta, const abcd_gaussians* grads,
                             abcd_gaussians* m, abcd_gaussians* v, const float lr[6],
                             float beta1, float beta2, float eps, int step);

/* One active-block step of Section 2 in one call: K2 abcd_project, K3-K4 abcd_bin_sort, K5
 * abcd_render_composite_fwd (out_rgba and state), K6-K8 abcd_backward with the loss against
 * gt_rgb (its gradient in the workspace) into grads, K9 abcd_adam_active.  The same as calling
 * those entry points in that order with these arguments; one call instead of six saves the
 * caller's per-call cost on a step of about thirty launches.  The first failing call's status
 * is returned (later ones are not made). */
abcd_status abcd_train_step(abcd_ctx* ctx, abcd_gaussians* theta, abcd_gaussians* grads,
                            abcd_gaussians* m, abcd_gaussians* v, const abcd_camera* cam,
                            const abcd_render_opts* opts, abcd_projected* proj, abcd_tiles* tiles,
                            const void* F, const void* B, int fb_dtype, const float* bg,
                            float* out_rgba, abcd_fwd_state* state, const float* gt_rgb,
                            float lambda_ssim, float* loss_out, const float lr[6], float beta1,
                            float beta2, float eps, int step);

/* K1. Depth-ordered over-compositing of cached per-partition renders into the foreground F and
 * background B of one camera (Section 2: the frozen partitions' stored renders, taken in the
 * camera's depth order, collapse into two RGBA images).  layers: host array of L device pointers to [H][W][4] premultiplied RGBA of
 * layer_dtype; order: host array of L indices, front to back; split: position in order of
 * the active partition (its layer is skipped and may be NULL), or L for "all in front".
 * F_out = fold over order[0 .. split), B_out = fold over order[split+1 .. L), each a left
 * fold of X over Y from transparent, accumulated in fp32 and rounded once to out_dtype.
 * L <= 256.  Either output may be NULL. */
abcd_status abcd_composite_cache(abcd_ctx* ctx, const void* const* layers, int L,
                                 int layer_dtype, const int* order, int split, int width,
                                 int height, void* F_out, void* B_out, int out_dtype);

/* Packed layers: the tile-sparse format of the cache (a lossless compression of the stored
 * renders of Section 2, which are transparent wherever their partition puts no Gaussian).
 * Over the 16x16-pixel tile grid of the image, tile_map[t] (int, [tiles]) is -1 for a tile
 * that is not stored (every pixel (0, 0, 0, 0)), else the index of its block in `packed`:
 * 16 x 16 fp16 RGBA pixels, row-major inside the tile (2 KB per block), blocks numbered in
 * tile order.  Pixels of a stored border tile that fall outside the image are unspecified. */

/* K10 into a packed layer: renders the active block alone (as abcd_render_composite_fwd's
 * refresh_f16, F = B = transparent) and stores the tiles whose list (from abcd_bin_sort) is
 * non-empty; a tile with an empty list renders (0, 0, 0, 0) exactly.  tile_map: device
 * [tiles] int; packed: device, room for one block per tile, 16-byte aligned; count: device int
 * receiving the number of stored tiles.  ABCD_ERR_INVALID_ARG for null or misaligned
 * buffers. */
abcd_status abcd_render_refresh_packed(abcd_ctx* ctx, const abcd_camera* cam,
                                       const abcd_render_opts* opts, const abcd_projected* proj,
                                       const abcd_tiles* tiles, int* tile_map, void* packed,
                                       int* count);

/* K10 for one camera in one call: abcd_project, abcd_bin_sort and
 * abcd_render_refresh_packed with these arguments, in that order (the first failing call's
 * status is returned). */
abcd_status abcd_refresh_layer(abcd_ctx* ctx, const abcd_gaussians* theta, const abcd_camera* cam,
                               const abcd_render_opts* opts, abcd_projected* proj,
                               abcd_tiles* tiles, int* tile_map, void* packed, int* count);

/* K1 over packed layers: the same folds as abcd_composite_cache (fp16 layers), with layer k
 * given by tile_maps[k] and packed[k] (host arrays of L device pointers; NULL at the active
 * position).  A tile a layer does not store is transparent for it, which leaves the fold
 * unchanged, so the result equals abcd_composite_cache on the decoded layers bit for bit;
 * only stored tiles are read. */
abcd_status abcd_composite_cache_packed(abcd_ctx* ctx, const int* const* tile_maps,
                                        const void* const* packed, int L, const int* order,
                                        int split, int width, int height, void* F_out,
                                        void* B_out, int out_dtype);

/* One side of K1 in pieces, for devices that cannot hold every frozen layer of a camera at once
 * (Section 2's memory hierarchy: the stored renders stay in host memory or on disk and pass
 * through a device buffer of fixed size).  acc_out = acc_in over layer 0 over layer 1 ... over
 * layer count-1 (packed layers as for abcd_composite_cache_packed, tile_maps[k] / packed[k] in
 * fold order; acc_in NULL: from transparent), fp32 premultiplied RGBA [H][W][4]; out16, if not
 * NULL, receives the fp16 (RNE) rounding of the result.  acc_in may equal acc_out.  The fp32
 * operations and their order are those of abcd_composite_cache_packed, so folding F's (or B's)
 * layers piece by piece into one accumulator and rounding at the end gives its F (B) bit for
 * bit.  count <= 256. */
abcd_status abcd_composite_fold_packed(abcd_ctx* ctx, const int* const* tile_maps,
                                       const void* const* packed, int count, int width,
                                       int height, const float* acc_in, float* acc_out,
                                       void* out16);

/* Visibility of the cached layers of one camera, for the visibility thresholds and occlusion
 * culling of camera-partition pairs that Section 4 proposes.  The layers are taken in `order`
 * (host, `count` distinct indices below L, front to back; a layer left out counts as absent).
 * For the layer at position k, with alpha_k its alpha and T_k the product of (1 - alpha) over
 * the layers before it:
 *   visible[order[k]]  = mean over the W x H pixels of alpha_k T_k (its share of the composite),
 *   coverage[order[k]] = mean of alpha_k (its image area, occluders ignored);
 * both 0 for layers not in the order.  Leaving a set D of layers out of the composite changes
 * every channel of every pixel by at most the sum over D of alpha_j T_j (premultiplied colours
 * at most alpha), so the sum of the dropped layers' visible shares bounds the mean error of
 * the culled composite.  layers: host array of L device pointers to fp16 [H][W][4]
 * premultiplied RGBA with alpha in [0, 1] (8-byte aligned; entries of layers not in the order
 * are not read and may be NULL); visible, coverage: device double [L] (coverage may be NULL),
 * overwritten.  The sums are exact in 24-bit fixed point per pixel value (result
 * independent of the order of the additions); they use the context's workspace (ABCD_ERR_WORKSPACE
 * without one).  L <= 256; ABCD_ERR_INVALID_ARG for a repeated or out-of-range index, a NULL
 * or misaligned layer or output. */
abcd_status abcd_layer_visibility(abcd_ctx* ctx, const void* const* layers, int L,
                                  const int* order, int count, int width, int height,
                                  double* visible, double* coverage);

/* abcd_layer_visibility over packed layers (tile_maps[k], packed[k] as for
 * abcd_composite_cache_packed); a tile a layer does not store is transparent. */
abcd_status abcd_layer_visibility_packed(abcd_ctx* ctx, const int* const* tile_maps,
                                         const void* const* packed, int L, const int* order,
                                         int count, int width, int height, double* visible,
                                         double* coverage);

/* The loss of abcd_loss without a context or workspace, for callers that cannot allocate
 * device memory: code running inside a host application that owns every device allocation
 * (its own pool or arena, with raw cudaMalloc forbidden), or a caller that must not allocate
 * between set-up and a latency-critical loop.  The paper has no counterpart; it exists only
 * for those callers.  Same arguments and results as abcd_loss, with an explicit stream.
 * Its scratch (per-CTA partial sums and a completion counter, about 512 KB) is a static
 * device array of this library, held by every GPU that loads the library until the process
 * exits; images may have at most 8192 x 4096 pixels (and 65536 CTAs, one per channel of a
 * 64x28-pixel tile), larger ones return ABCD_ERR_WORKSPACE before any launch.  The first call on a device (made with
 * that device current) loads the library's device code there and looks up the array's
 * address, so make it before any stream capture; later calls look the address up again (a
 * host-side table read), so a device reset never leaves a stale address.  All calls on a device share
 * the array: calls whose kernels overlap on the GPU race and give wrong losses, so order them
 * (one stream, or events).  The counter is cleared at the start of every call.  Returns
 * ABCD_ERR_INVALID_ARG for bad pointers, sizes or lambda, ABCD_ERR_CUDA if the address lookup,
 * the counter's clear or the launch fails (the launch's own status; earlier errors of other
 * work are not reported here).  loss_out and dL_dout may each be NULL. */
abcd_status abcd_loss_static(void* cuda_stream, const float* out_rgba, const float* gt_rgb,
                             int width, int height, float lambda_ssim, float* loss_out,
                             float* dL_dout);

/* ---- host tier of the layer cache (Section 2: the stored renders of the frozen
 * partitions are kept in host memory and brought to the GPU when a stage composites them;
 * refreshed renders go back).  Copies run on two copy streams of the context (host to
 * device, device to host) and overlap the kernels on its stream; slots (e.g. one per camera)
 * order them.  Host buffers should be pinned (cudaHostAlloc / cudaHostRegister); pageable
 * memory makes a copy synchronous.  One cudaMemcpyAsync per call. ------------------------ */

#define ABCD_MAX_CACHE_SLOTS 4096

/* Queues a copy of `bytes` bytes from host_src (host) to dev_dst (device) for `slot`
 * (0 <= slot < ABCD_MAX_CACHE_SLOTS).  It starts after the work that was queued on the
 * context's stream before the slot's last abcd_cache_release (at once if there was none), so
 * a slot's device data is not overwritten while a kernel still reads it.  Returns
 * ABCD_ERR_INVALID_ARG for a null pointer, bytes == 0 or a bad slot (nothing queued),
 * ABCD_ERR_CUDA if a copy or an event fails. */
abcd_status abcd_cache_fetch(abcd_ctx* ctx, int slot, const void* host_src, void* dev_dst,
                             size_t bytes);

/* Makes the context's stream wait until every fetch and store of `slot` queued so far is
 * done (nothing to wait for if there was none).  ABCD_ERR_INVALID_ARG for a bad slot. */
abcd_status abcd_cache_wait(abcd_ctx* ctx, int slot);

/* Marks the end of the reads of `slot`'s device data: later fetches of the slot start after
 * the work queued on the context's stream so far.  ABCD_ERR_INVALID_ARG for a bad slot. */
abcd_status abcd_cache_release(abcd_ctx* ctx, int slot);

/* Queues a copy of `bytes` bytes from dev_src (device) to host_dst (host) for `slot` that
 * starts after the work queued on the context's stream so far (a refreshed render going back
 * to the host tier while the next stage computes); a later abcd_cache_wait(slot) also waits
 * for it, so the device data is not rewritten before it has left.  ABCD_ERR_INVALID_ARG for a
 * null pointer, bytes == 0 or a bad slot. */
abcd_status abcd_cache_store(abcd_ctx* ctx, int slot, const void* dev_src, void* host_dst,
                             size_t bytes);

/* Waits until the context's queued fetches and stores are done (abcd_sync waits for its
 * compute stream only). */
abcd_status abcd_cache_sync(abcd_ctx* ctx);

/* ---- instrumentation: the arithmetic peaks the roofline fractions are taken against ----- */

typedef struct {
  int sms;                   /* multiprocessors, read from the device */
  double clock_mhz_nominal;  /* the device's reported SM clock (the runs take whatever clock
                                the GPU is at; nothing is locked or changed) */
  double ffma_tflops;        /* fp32 FMA, scalar FFMA, 2 flops per FMA */
  double ffma2_tflops;       /* fp32 FMA through the packed two-lane FFMA2 */
  double ex2_tops;           /* ex2.approx.ftz.f32 (MUFU) results per second, 1e12 */
  double ms_ffma, ms_ffma2, ms_ex2;   /* best timed launch of each kernel */
} abcd_alu_peaks;

/* Measures fp32 FMA and ex2.approx throughput on `device` with three short kernels of
 * independent dependency chains over 4 CTAs of 256 threads per SM (about 10 ms each, timed with
 * CUDA events on a private stream after a warm-up launch; best of five).  Synchronous; allocates
 * nothing.  ABCD_ERR_CUDA if a launch or event fails. */
abcd_status abcd_measure_alu_peaks(int device, abcd_alu_peaks* out);

/* ---- visible camera-partition pairs (Section 2 caches renders of the visible pairs and
 * trains a block on the cameras observing its partition; Section 3 speaks of the cameras left
 * after frustum filtering) ------------------------------------------------------------------ */

/* The axis-aligned box holding every Gaussian's 3-sigma ellipsoid of theta: box[0..2] lowest
 * x, y, z, box[3..5] highest (device float [6], written; for Sigma = R(q) diag(exp(2 log_scale))
 * R(q)^T the ellipsoid reaches mean_k +- 3 sqrt(Sigma_kk) along axis k, widened by 1e-6 relative
 * for fp32 rounding).  An empty block gives lowest > highest.  One CTA (a per-stage call). */
abcd_status abcd_block_bounds(abcd_ctx* ctx, const abcd_gaussians* theta, float* box);

/* Whether a partition whose extent is the box (host double [6], as abcd_block_bounds; take the
 * union with the cell) may be seen by the camera: the camera-space view frustum is
 * {z >= near_z, |x| <= gx z, |y| <= gy z}, gx = guard * (width / 2) / fx, gy likewise; the
 * pair is not visible (*visible = 0) only when the whole box lies outside one of those five
 * half-spaces, so a box that meets the frustum is never culled (a few boxes near the frustum's
 * edges that miss it are kept).  An empty box is not visible.  Host only. */
abcd_status abcd_pair_visible(const abcd_camera* cam, const abcd_render_opts* opts,
                              const double box[6], int* visible);

/* ---- host-side partition logic (Section 2: regular grid, assignment by mean) --------- */

/* cell[i] = linear id (i + gx (j + gy k)) of the grid cell holding means[i] (host array,
 * [n][3] float), clamped into the grid. */
abcd_status abcd_assign_cells(const float* means_host, int n, const double origin[3],
                              double side, const int dims[3], int* cell);

/* Front-to-back order of the frozen partitions seen from campos and the split at the active
 * partition.  A cell's key is its Manhattan distance (in cells) from the camera's cell (not
 * clamped into the grid); along any ray the key grows strictly from cell to cell, so every
 * cell with a smaller key than the active one that shares a ray with it lies in front.
 * front/back: capacity for gx*gy*gz entries; ascending (key, id); equal keys go behind. */
abcd_status abcd_partition_split(const int dims[3], const double origin[3], double side,
                                 const double campos[3], int active, int* front, int* n_front,
                                 int* back, int* n_back);

#ifdef __cplusplus
}
#endif
#endif
