/* CPU oracle for the ABCD active-block step -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, per-pixel / per-Gaussian fp64 implementation of what the ABCD hot path
 * computes: 3D Gaussian Splatting projection with spherical-harmonic colour, tile binning
 * with a stable (tile, depth) sort, front-to-back alpha blending of the active block,
 * over-compositing with the cached foreground F and background B (Section 2: the frozen
 * blocks in front of / behind the active partition collapse into two RGBA images by
 * associativity of alpha compositing), the L1 + D-SSIM reconstruction loss, the gradient
 * back into the active block only, Adam, and the depth-ordered compositing of cached
 * per-partition renders into F and B (Section 2).
 * The renderer formulas are those of 3D Gaussian Splatting, which the paper instantiates
 * by citation (Section 1, last paragraph); Section 2 fixes the compositing structure.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may load this
 * library.  It shares no code with the CUDA path (paper_2608_27735_gb300/csrc).
 *
 * Parity status per function (what pins it; see tests/test_oracle_*.py):
 *   orc_project            single-Gaussian closed form, SH vs scipy, brute-force rect
 *   orc_project_backward   central finite differences (fp64)
 *   orc_tile_lists         brute-force per-tile scan + Python sort; listing rule against the
 *                          square rule (identical images) and dense box sampling
 *   orc_render_pixel/image closed form, invariants, associativity identity
 *   orc_backward_pixel/... central finite differences (fp64), incl. the F/B alpha term
 *   orc_composite_layers   constant-layer closed form, split invariance
 *   orc_layer_visibility   telescoping identity against the composite's alpha, opaque and
 *                          single-layer cases, the culling error bound
 *   orc_loss               SSIM(x,x)=1, scipy 2-D correlation, finite differences
 *   orc_adam               first-step closed form, hand-computed second step
 *   orc_assign_cells / orc_partition_split   brute-force ray sampling of the depth order
 *   orc_block_bounds       sampled points of every 3-sigma ellipsoid inside the box, its
 *                          faces touched
 *   orc_pair_visible       dense sampling of boxes: a box with a sampled point inside the
 *                          frustum is never culled; closed-form cases
 */
#ifndef ABCD_ORACLE_H
#define ABCD_ORACLE_H

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  double R[9];              /* world -> camera rotation, row-major; x right, y down, z fwd */
  double t[3];              /* world -> camera translation */
  double fx, fy, cx, cy;    /* pinhole intrinsics, pixels; pixel (i, j) covers [i, i+1) */
  int width, height;
} orc_camera;

typedef struct {
  double near_z;            /* cull Gaussians with camera z <= near_z (0.2) */
  double dilation;          /* added to the 2-D covariance diagonal (0.3) */
  double guard;             /* Jacobian evaluated with x/z clamped to guard*tan(fov/2) (1.3) */
  double alpha_max;         /* alpha clamp (0.99) */
  double alpha_min;         /* skip contributions with alpha below this (1/255) */
  double t_min;             /* stop before a Gaussian that would take T below this (1e-4) */
  int tile;                 /* tile edge in pixels (16) */
} orc_opts;

typedef struct {
  const double* means;          /* [n][3] */
  const double* log_scales;     /* [n][3] */
  const double* quats;          /* [n][4] (w, x, y, z), not necessarily unit */
  const double* opacity_logits; /* [n] */
  const double* sh;             /* [n][D][3], D = (deg+1)^2, index l*l + l + m */
  int n;
  int sh_degree;                /* 0..3 */
} orc_gaussians;

typedef struct {               /* screen-space splats the per-pixel renderer reads */
  int n;
  const double* uv;            /* [n][2] */
  const double* conic;         /* [n][3] */
  const double* opacity;       /* [n] */
  const double* rgb;           /* [n][3] */
} orc_splats;

typedef struct {
  int* visible;             /* [n] 1 if z > near and the tile rectangle is non-empty */
  double* depth;            /* [n] camera-space z */
  unsigned* depth_key;      /* [n] IEEE bits of the fp32 depth ((R6*x + R7*y) + R8*z) + t2 */
  double* uv;               /* [n][2] pixel-space mean */
  double* conic;            /* [n][3] (a, b, c) of the inverse 2-D covariance [[a,b],[b,c]] */
  double* opacity;          /* [n] */
  double* rgb;              /* [n][3] colour, clamped at 0 */
  double* rgb_raw;          /* [n][3] colour before the clamp */
  double* eig;              /* [n][2] eigenvalues (max, min) of the dilated 2-D covariance */
  double* radius_exact;     /* [n] 3*sqrt(lambda_max') with the 0.1 floor of 3DGS */
  int* radius;              /* [n] ceil(radius_exact) */
  int* rect;                /* [n][4] tile rectangle x0, y0, x1, y1 (half-open) */
  double* view_tan;         /* [n][2] x/z and y/z (to locate the guard clamp) */
} orc_projected;


/* Uncertainty model used only to REPORT decisions of the blend loop that lie so close to
 * their threshold that an fp32 implementation may take either branch.  NULL = no events. */
typedef struct {
  const double* m_uv;          /* [n][2] absolute uncertainty of u, v (pixels) */
  const double* m_conic;       /* [n] relative uncertainty of the conic */
  double k_arith;              /* relative rounding of sigma w.r.t. its absolute terms */
  double eps_alpha;            /* relative error of exp / opacity in alpha */
  double eps_step;             /* relative rounding per transmittance update */
} orc_margins;

enum { ORC_EV_SKIP = 1, ORC_EV_TERM = 2, ORC_EV_CLAMP = 3 };

void orc_default_opts(orc_opts* o);

int orc_project(const orc_gaussians* g, const orc_camera* cam, const orc_opts* o,
                orc_projected* out);

/* Gradient of sum_k <grad2d[k], (u, v, a, b, c, opacity, r, g, b)_k> w.r.t. the parameters
 * (forward-mode dual numbers through the projection definition). Outputs overwritten. */
int orc_project_backward(const orc_gaussians* g, const orc_camera* cam, const orc_opts* o,
                         const double* grad2d /*[n][9]*/, double* d_means, double* d_log_scales,
                         double* d_quats, double* d_opacity_logits, double* d_sh);

/* Stable sort of (tile, depth_key) over all visible Gaussians emitted in id order.
 * offsets has n_tiles+1 entries; ids has capacity entries.  Returns K (or -K-1 if
 * K > capacity; nothing is written then).
 * Listing rule: tile t of Gaussian i's rectangle is kept when s (uv, conic, opacity) is NULL,
 * else only if the Gaussian can reach alpha >= alpha_min on t: o >= alpha_min and the minimum
 * of sigma over the box of t's pixel centres [16 tx + 0.5, 16 tx + 15.5] x [...] is
 * <= ln(o / alpha_min).  Dropped entries are skipped by every pixel of t anyway.
 * With margin_rel or margin_abs non-zero (the renderer's listing reading, R1b), the test is
 * m / ln 2 <= (thr (1 + margin_rel) + margin_abs) (1 + margin_rel), thr = log2(o / alpha_min):
 * a superset of the exact rule's lists whose extra entries every pixel of their tile skips. */
long long orc_tile_lists(int n, const int* visible, const int* rect, const unsigned* depth_key,
                         int tiles_x, int tiles_y, long long* offsets, int* ids,
                         long long capacity, const orc_splats* s, double alpha_min, int tile,
                         double margin_rel, double margin_abs);

/* Minimum of sigma(d) = 1/2 (a dx^2 + c dy^2) + b dx dy over the box [X0, X1] x [Y0, Y1]
 * (convex: 0 if the box holds d = 0, else the least value on its four edges). */
double orc_box_min_sigma(const double* conic, double X0, double X1, double Y0, double Y1);

/* One pixel: front-to-back blend of list[0..len) then F over (A over B), + (1-out.a)*bg.
 * F, B: 4 doubles (premultiplied RGBA) or NULL (transparent).  toggles: n_toggles pairs
 * (gaussian id, ORC_EV_*) inverting that decision.  Events of this run are reported. */
int orc_render_pixel(const orc_splats* s, const int* list, int len, int px, int py,
                     const orc_opts* o, const double* F, const double* B, const double* bg,
                     const int* toggles, int n_toggles, const orc_margins* mg,
                     double* out4, double* A4, double* T_final, int* n_used,
                     int* ev, int max_ev, int* n_ev);

/* Whole image over per-tile lists.  F, B: [H][W][4] or NULL.  Events: up to max_ev per
 * pixel into ev[P][max_ev][2], counts into n_ev[P] (all may be NULL). */
int orc_render_image(const orc_splats* s, const long long* offsets, const int* ids,
                     int width, int height, const orc_opts* o, const double* F,
                     const double* B, const double* bg, const orc_margins* mg,
                     double* out, double* A, double* T_final, int* n_used,
                     int* ev, int max_ev, int* n_ev);

/* Backward of one pixel given G = dL/d(final rgb) (3 values): accumulates the gradient
 * w.r.t. (u, v, a, b, c, opacity, r, g, b) of every contributing Gaussian into grad2d. */
int orc_backward_pixel(const orc_splats* s, const int* list, int len, int px, int py,
                       const orc_opts* o, const double* F, const double* B, const double* bg,
                       const int* toggles, int n_toggles, const double* G, double* grad2d);

int orc_backward_image(const orc_splats* s, const long long* offsets, const int* ids,
                       int width, int height, const orc_opts* o, const double* F,
                       const double* B, const double* bg, const double* G /*[H][W][3]*/,
                       double* grad2d /*[n][9], overwritten*/);

/* orc_backward_image restricted to the pixels listed (linear indices, ascending); equal to it
 * when G is zero at every other pixel.  Returns 1 for an index outside the image. */
int orc_backward_pixels(const orc_splats* s, const long long* offsets, const int* ids,
                        int width, int height, const orc_opts* o, const double* F,
                        const double* B, const double* bg, const double* G,
                        const int* pixels, int n_pixels, double* grad2d);

/* Left fold of X over Y = X + (1 - X.a) * Y over layers[order[k]] for k in the given
 * sequence, starting from transparent.  layers: [L][P][4]. out: [P][4]. */
int orc_composite_layers(int n_pixels, const double* layers, const int* order, int count,
                         double* out);

/* Visibility of each layer of one camera's depth order (Section 4: visibility thresholds and
 * occlusion culling of camera-partition pairs).  For the layer at position k of the order,
 * with alpha_k its alpha and T_k the product of (1 - alpha) over the layers before it:
 * visible[order[k]] = mean over pixels of alpha_k T_k, coverage[order[k]] = mean of alpha_k;
 * layers not listed get 0.  layers: [L][P][4]; order: count distinct indices below L.
 * Returns 1 for a repeated or out-of-range index. */
int orc_layer_visibility(int n_pixels, int n_layers, const double* layers, const int* order,
                         int count, double* visible, double* coverage);

/* (1 - lam) * mean|x - y| + lam * (1 - mean SSIM(x, y)), 11x11 Gaussian window (sigma 1.5),
 * zero padding, C1 = 0.01^2, C2 = 0.03^2; x, y: [H][W][3].  grad (may be NULL) = dL/dx. */
int orc_loss(int width, int height, const double* x, const double* y, double lam,
             double* loss, double* grad);

/* SSIM map only (for pins): [H][W][3]. */
int orc_ssim_map(int width, int height, const double* x, const double* y, double* map);

/* torch-style Adam with bias correction on one parameter group (step is 1-based). */
int orc_adam(long long n, double* theta, const double* grad, double* m, double* v, double lr,
             double beta1, double beta2, double eps, int step);

/* Partition of a Gaussian = grid cell of its mean, clamped into the grid;
 * linear id = i + gx * (j + gy * k). */
int orc_assign_cells(int n, const double* means, const double* origin, double side,
                     const int* dims, int* cell);

/* Front-to-back order of the frozen partitions for a camera at campos and the split at the
 * active partition: key(j) = Manhattan distance between cell j and the camera's
 * (unclamped) cell; ascending key, ties by id; front = key < key(active), back = the rest
 * (active excluded).  Returns 0; nf / nb receive the counts. */
int orc_partition_split(const int* dims, const double* origin, double side,
                        const double* campos, int active, int* front, int* nf, int* back,
                        int* nb);

/* Axis-aligned box of the 3-sigma ellipsoids of g: box[0..2] lowest, box[3..5] highest corner
 * (half-width along axis k: 3 sqrt(Sigma_kk), Sigma = R(q) diag(exp(2 log_scale)) R(q)^T). */
int orc_block_bounds(const orc_gaussians* g, double* box);

/* Whether the box may be seen by the camera (reading R14): it is culled only when all eight
 * corners lie, in camera space, on the outer side of one bounding plane of the view frustum
 * {z >= near_z, |x| <= gx z, |y| <= gy z}, gx = guard * (width / 2) / fx (gy likewise). */
int orc_pair_visible(const orc_camera* cam, const orc_opts* o, const double* box, int* visible);

/* Real spherical harmonic Y_lm (Condon-Shortley phase) at a unit direction (for pins). */
double orc_sh_basis(int l, int m, double x, double y, double z);

#ifdef __cplusplus
}
#endif
#endif
