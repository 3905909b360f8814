// Context, workspace, status word and host-side partition logic of libabcd.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <vector>

#include "abcd_internal.cuh"

namespace abcd {

abcd_status fail(abcd_ctx* ctx, abcd_status code, const char* fmt, ...) {
  if (ctx) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(ctx->err, sizeof ctx->err, fmt, ap);
    va_end(ap);
  }
  return code;
}

abcd_status check_launch(abcd_ctx* ctx, const char* what) {
  ctx->launches++;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  return ABCD_OK;
}

abcd_status check_launch(abcd_ctx* ctx, const char* what, cudaError_t launched) {
  if (launched != cudaSuccess) {
    ctx->launches++;
    (void)cudaGetLastError();
    return fail(ctx, ABCD_ERR_CUDA, "%s: %s", what, cudaGetErrorString(launched));
  }
  return check_launch(ctx, what);
}

bool has_workspace(const abcd_ctx* ctx) { return ctx && ctx->ws_base != nullptr; }

// Zeroes `words` 4-byte words at p (4-byte aligned): 16-byte stores over the aligned body, 4-byte
// ones around it.  A kernel rather than a memset: launched with programmatic serialisation, it
// keeps the launches of a call overlapping the tails of the kernels before them.
__global__ void __launch_bounds__(256) zero_kernel(unsigned* p, long long words) {
  pdl_prologue();
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long stride = (long long)gridDim.x * blockDim.x;
  const long long head = min((long long)(((16u - ((uintptr_t)p & 15u)) & 15u) / 4u), words);
  const long long body = (words - head) / 4;
  for (long long i = tid; i < head; i += stride) p[i] = 0u;
  uint4* q = reinterpret_cast<uint4*>(p + head);
  for (long long i = tid; i < body; i += stride) q[i] = make_uint4(0u, 0u, 0u, 0u);
  for (long long i = head + 4 * body + tid; i < words; i += stride) p[i] = 0u;
}

abcd_status zero_async(abcd_ctx* ctx, void* p, size_t bytes, const char* what) {
  if (bytes == 0) return ABCD_OK;
  if (((uintptr_t)p & 3) || (bytes & 3)) {
    const cudaError_t e = cudaMemsetAsync(p, 0, bytes, ctx->stream);
    return e == cudaSuccess ? ABCD_OK : fail(ctx, ABCD_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  }
  const long long words = (long long)(bytes / 4);
  const long long blocks = std::min<long long>((words / 4 + 255) / 256 + 1, 4LL * ctx->num_sms);
  return check_launch(ctx, what, launch_pdl(zero_kernel, dim3((unsigned)blocks), dim3(256), 0,
                                            ctx->stream, (unsigned*)p, words));
}

cudaError_t ensure_smem(abcd_ctx* ctx, const void* fn, size_t bytes) {
  if (bytes <= 48 * 1024) return cudaSuccess;
  int slot = -1;
  for (int i = 0; i < 16; ++i) {
    if (ctx->smem_fn[i] == fn) { slot = i; break; }
    if (!ctx->smem_fn[i] && slot < 0) slot = i;
  }
  if (slot >= 0 && ctx->smem_fn[slot] == fn && ctx->smem_set[slot] >= (int)bytes) return cudaSuccess;
  int prev = 0;
  cudaGetDevice(&prev);
  if (prev != ctx->device) cudaSetDevice(ctx->device);
  const cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (prev != ctx->device) cudaSetDevice(prev);
  if (e == cudaSuccess && slot >= 0) { ctx->smem_fn[slot] = fn; ctx->smem_set[slot] = (int)bytes; }
  return e;
}

Opts make_opts(const abcd_render_opts* o) {
  Opts r;
  r.near_z = o ? o->near_z : 0.2f;
  r.dilation = o ? o->dilation : 0.3f;
  r.guard = o ? o->guard : 1.3f;
  r.alpha_max = o ? o->alpha_max : 0.99f;
  r.alpha_min = o ? o->alpha_min : 1.0f / 255.0f;
  r.t_min = o ? o->t_min : 1e-4f;
  return r;
}

Cam make_cam(const abcd_camera* c, const abcd_render_opts* o) {
  Cam k;
  for (int i = 0; i < 9; ++i) k.R[i] = c->R[i];
  for (int i = 0; i < 3; ++i) k.t[i] = c->t[i];
  k.fx = c->fx; k.fy = c->fy; k.cx = c->cx; k.cy = c->cy;
  for (int j = 0; j < 3; ++j) {
    double s = 0.0;
    for (int i = 0; i < 3; ++i) s -= (double)c->R[3 * i + j] * (double)c->t[i];
    k.campos[j] = (float)s;
  }
  const float guard = o ? o->guard : 1.3f;
  k.limx = guard * (0.5f * (float)c->width / c->fx);
  k.limy = guard * (0.5f * (float)c->height / c->fy);
  k.width = c->width; k.height = c->height;
  k.tiles_x = (c->width + kTile - 1) / kTile;
  k.tiles_y = (c->height + kTile - 1) / kTile;
  return k;
}

// Normalisation of the real SH basis: Y_l^0 = K_l^0 P_l(z); for m != 0,
// Y_l^(+-m) = sqrt2 K_l^m (-1)^m P_l^(m)(z) Re/Im (x + i y)^m with
// K_l^m = sqrt((2l + 1)/(4 pi) (l - m)!/(l + m)!).  The kernels multiply k[l*l+l+m] by the
// Legendre derivative polynomial and the Cartesian factor.
void sh_constants(SHConst* out) {
  auto fact = [](int n) { double r = 1; for (int i = 2; i <= n; ++i) r *= i; return r; };
  const double pi = 3.14159265358979323846;
  for (int l = 0; l <= 3; ++l)
    for (int m = -l; m <= l; ++m) {
      const int am = m < 0 ? -m : m;
      const double K = std::sqrt((2.0 * l + 1.0) / (4.0 * pi) * fact(l - am) / fact(l + am));
      const double k = (m == 0) ? K : std::sqrt(2.0) * K * ((am & 1) ? -1.0 : 1.0);
      out->k[l * l + l + m] = (float)k;
    }
}

}  // namespace abcd

using namespace abcd;

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

extern "C" {

abcd_status abcd_create(abcd_ctx** out, int device, void* stream) {
  if (!out) return ABCD_ERR_INVALID_ARG;
  *out = nullptr;
  abcd_ctx* ctx = new (std::nothrow) abcd_ctx();
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  ctx->device = device;
  ctx->stream = (cudaStream_t)stream;
  int prev = 0;
  cudaGetDevice(&prev);
  cudaError_t e = cudaSetDevice(device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, device);
  // side stream for work that runs beside the main stream inside one call (fork / join)
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&ctx->side, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_fork, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_join, cudaEventDisableTiming);
  cudaSetDevice(prev);
  if (e != cudaSuccess) {
    abcd_destroy(ctx);
    return ABCD_ERR_CUDA;
  }
  ctx->radix_blocks = std::min(kMaxRadixBlocks, 2 * ctx->num_sms);
  sh_constants(&ctx->sh);
  *out = ctx;
  return ABCD_OK;
}

abcd_status abcd_destroy(abcd_ctx* ctx) {
  if (!ctx) return ABCD_OK;
  cache_destroy(ctx);
  if (ctx->ev_fork) cudaEventDestroy(ctx->ev_fork);
  if (ctx->ev_join) cudaEventDestroy(ctx->ev_join);
  if (ctx->side) cudaStreamDestroy(ctx->side);
  delete ctx;
  return ABCD_OK;
}

abcd_status abcd_set_stream(abcd_ctx* ctx, void* stream) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  ctx->stream = (cudaStream_t)stream;
  return ABCD_OK;
}

static size_t layout(char* base, int max_g, long long max_pairs, long long max_pixels,
                     Workspace* ws) {
  size_t off = 0;
  auto take = [&](size_t bytes) { char* p = base ? base + off : nullptr; off += align256(bytes); return p; };
  Workspace w;
  w.status = (unsigned*)take(256);
  w.dsort[0] = (unsigned long long*)take(8ull * (size_t)max_g);
  w.dsort[1] = (unsigned long long*)take(8ull * (size_t)max_g);
  w.pairs[0] = (unsigned long long*)take(8ull * (size_t)max_pairs);
  w.pairs[1] = (unsigned long long*)take(8ull * (size_t)max_pairs);
  w.os_gh = (unsigned*)take(4ull * 2 * 4 * kRadixBins);
  w.os_ctr = (unsigned*)take(256);
  // look-back words: a sort tile holds at least 1024 items; the run placement publishes one
  // word per tile column for each chunk of 512 runs (runs <= pairs) and row
  w.os_tiles = std::max<long long>((std::max<long long>(max_pairs, max_g) + 1023) / 1024,
                                   (max_pairs + 511) / 512 + kMaxRunRows) + 1;
  w.os_state = (unsigned long long*)take(8ull * kRadixBins * (size_t)w.os_tiles);
  w.rects = (int4*)take(16ull * (size_t)max_g);
  w.counts = (unsigned*)take(4ull * (size_t)max_g);
  w.row_runs = (unsigned*)take(4ull * kMaxRunRows);
  w.n_runs = (long long*)take(8);
  w.diff_bytes = 4ull * kMaxDiffCells;
  w.diff = (int*)take(w.diff_bytes);
  w.block_sums = (unsigned long long*)take(8ull * (kMaxRadixBlocks + 1));
  w.grad2d = (float*)take(4ull * 9 * (size_t)max_g);
  w.dl_dout = (float*)take(4ull * 3 * (size_t)max_pixels);
  w.loss_partials = (float*)take(4ull * 2 * kMaxLossBlocks);
  w.ssim_ab = (float2*)take(8ull * 3 * (size_t)max_pixels);
  w.ssim_c = (float*)take(4ull * 3 * (size_t)max_pixels);
  w.max_tiles = max_order_tiles(max_pixels);
  w.tile_order = (unsigned*)take(4ull * (size_t)w.max_tiles);
  w.ck_cap = (int)std::max<long long>(1024, max_pixels / 128);
  w.ckpt = (float4*)take(16ull * 64 * (size_t)w.ck_cap);
  w.ck_items = (uint4*)take(16ull * (size_t)w.ck_cap);
  w.ck_count = (unsigned*)take(256);
  w.ck_first = (unsigned*)take(4ull * 4 * (size_t)w.max_tiles);
  w.vis_sums = (unsigned long long*)take(8ull * kVisSumCopies * 2 * kMaxLayers);
  w.vis_ticket = (unsigned*)take(256);
  if (ws) *ws = w;
  return off;
}

abcd_status abcd_workspace_size(int max_gaussians, long long max_pairs, long long max_pixels,
                                size_t* bytes) {
  if (!bytes || max_gaussians < 0 || max_pairs < 0 || max_pixels < 0) return ABCD_ERR_INVALID_ARG;
  *bytes = layout(nullptr, max_gaussians, max_pairs, max_pixels, nullptr);
  return ABCD_OK;
}

abcd_status abcd_set_workspace(abcd_ctx* ctx, void* ptr, size_t bytes, int max_gaussians,
                               long long max_pairs, long long max_pixels) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!ptr || ((uintptr_t)ptr & 255)) return fail(ctx, ABCD_ERR_INVALID_ARG, "workspace must be a 256-byte aligned device pointer");
  if (max_gaussians < 0 || max_pairs < 0 || max_pixels < 0) return fail(ctx, ABCD_ERR_INVALID_ARG, "negative workspace limits");
  const size_t need = layout(nullptr, max_gaussians, max_pairs, max_pixels, nullptr);
  if (bytes < need) return fail(ctx, ABCD_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", bytes, need);
  ctx->ws_base = (char*)ptr;
  ctx->ws_bytes = bytes;
  ctx->max_g = max_gaussians;
  ctx->max_pairs = max_pairs;
  ctx->max_pixels = max_pixels;
  layout(ctx->ws_base, max_gaussians, max_pairs, max_pixels, &ctx->ws);
  cudaError_t e = cudaMemsetAsync(ctx->ws.status, 0, 256, ctx->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->ws.os_ctr, 0, 256, ctx->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->ws.vis_sums, 0, 8ull * kVisSumCopies * 2 * kMaxLayers, ctx->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(ctx->ws.vis_ticket, 0, 256, ctx->stream);

  if (e == cudaSuccess)
    e = cudaMemsetAsync(ctx->ws.os_state, 0, 8ull * kRadixBins * (size_t)ctx->ws.os_tiles, ctx->stream);
  ctx->os_epoch = 0;
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "clearing status: %s", cudaGetErrorString(e));
  return ABCD_OK;
}

abcd_status abcd_clear_status(abcd_ctx* ctx) {
  if (!has_workspace(ctx)) return ABCD_ERR_WORKSPACE;
  cudaError_t e = cudaMemsetAsync(ctx->ws.status, 0, 8, ctx->stream);
  return e == cudaSuccess ? ABCD_OK : fail(ctx, ABCD_ERR_CUDA, "clear status: %s", cudaGetErrorString(e));
}

abcd_status abcd_sync(abcd_ctx* ctx) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "stream: %s", cudaGetErrorString(e));
  if (!has_workspace(ctx)) return ABCD_OK;
  unsigned word = 0;
  e = cudaMemcpy(&word, ctx->ws.status, sizeof word, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "status read: %s", cudaGetErrorString(e));
  for (int code = 1; code < 32; ++code)
    if (word & (1u << code)) return fail(ctx, (abcd_status)code, "device reported status %d", code);
  return ABCD_OK;
}

const char* abcd_last_error(const abcd_ctx* ctx) { return ctx ? ctx->err : "null context"; }

abcd_status abcd_set_wait_limit(abcd_ctx* ctx, unsigned polls) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  ctx->wait_limit = polls;
  return ABCD_OK;
}

abcd_status abcd_test_withhold_lookback(abcd_ctx* ctx, long long tile) {
  if (!ctx || tile < -1) return ABCD_ERR_INVALID_ARG;
  ctx->withhold_tile = tile;
  return ABCD_OK;
}

long long abcd_launch_count(const abcd_ctx* ctx) { return ctx ? ctx->launches : 0; }

abcd_status abcd_assign_cells(const float* means, int n, const double origin[3], double side,
                              const int dims[3], int* cell) {
  if (n < 0 || (n > 0 && (!means || !cell)) || !origin || !dims || !(side > 0)) return ABCD_ERR_INVALID_ARG;
  for (int k = 0; k < 3; ++k)
    if (dims[k] <= 0) return ABCD_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    int c[3];
    for (int k = 0; k < 3; ++k) {
      const double f = std::floor(((double)means[3 * i + k] - origin[k]) / side);
      c[k] = (int)std::min<double>(std::max<double>(f, 0.0), dims[k] - 1);
    }
    cell[i] = c[0] + dims[0] * (c[1] + dims[1] * c[2]);
  }
  return ABCD_OK;
}

abcd_status abcd_partition_split(const int dims[3], const double origin[3], double side,
                                 const double campos[3], int active, int* front, int* n_front,
                                 int* back, int* n_back) {
  if (!dims || !origin || !campos || !front || !back || !n_front || !n_back || !(side > 0))
    return ABCD_ERR_INVALID_ARG;
  const long long total = (long long)dims[0] * dims[1] * dims[2];
  if (dims[0] <= 0 || dims[1] <= 0 || dims[2] <= 0 || active < 0 || active >= total)
    return ABCD_ERR_INVALID_ARG;
  long long cam_cell[3];
  for (int k = 0; k < 3; ++k) cam_cell[k] = (long long)std::floor((campos[k] - origin[k]) / side);
  std::vector<std::pair<long long, int>> keyed((size_t)total);
  for (int id = 0; id < total; ++id) {
    const long long ijk[3] = {id % dims[0], (id / dims[0]) % dims[1], id / (dims[0] * dims[1])};
    long long d = 0;
    for (int k = 0; k < 3; ++k) d += std::llabs(ijk[k] - cam_cell[k]);
    keyed[id] = {d, id};
  }
  const long long key_active = keyed[active].first;
  std::sort(keyed.begin(), keyed.end());
  int nf = 0, nb = 0;
  for (const auto& e : keyed) {
    if (e.second == active) continue;
    if (e.first < key_active) front[nf++] = e.second;
    else back[nb++] = e.second;
  }
  *n_front = nf;
  *n_back = nb;
  return ABCD_OK;
}

}  // extern "C"
