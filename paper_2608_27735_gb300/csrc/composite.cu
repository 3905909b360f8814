// K1: depth-ordered over-compositing of cached per-partition RGBA renders into F and B.
// Section 2 builds, per camera, the foreground and background images from the stored renders
// of the frozen partitions in the camera's depth order; by associativity of 'over' the frozen
// blocks in front of the active partition collapse into F, those behind it into B.
//
// Pure streaming work: every layer is read once (16-byte streaming loads, evict-first), the
// accumulator stays in registers across layers, F and B are written once.  Four layers are
// loaded before they are folded so each thread keeps 64 bytes in flight.  The grid is a
// multiple of the SM count and strides over pixel pairs.
#include "abcd_internal.cuh"

namespace abcd {
namespace {

struct LayerTable {
  const void* p[kMaxLayers];   // front layers in order, then back layers in order
};

__device__ __forceinline__ void unpack_h8(uint4 r, float* f) {
  const unsigned w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float2 v = __half22float2(*reinterpret_cast<const __half2*>(&w[k]));
    f[2 * k] = v.x;
    f[2 * k + 1] = v.y;
  }
}

__device__ __forceinline__ void unpack_h4(uint2 r, float* f) {
  const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&r.x));
  const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&r.y));
  f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
}

// acc (premultiplied RGBA x PIX pixels) = acc over layer
template <int PIX>
__device__ __forceinline__ void fold(float* acc, const float* L) {
#pragma unroll
  for (int q = 0; q < PIX; ++q) {
    const float k = 1.f - acc[4 * q + 3];
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[4 * q + c] = __fmaf_rn(k, L[4 * q + c], acc[4 * q + c]);
  }
}

// Loads PIX pixels (4 channels each) of layer `ptr` at pixel group g into f.
template <int PIX, bool F16>
__device__ __forceinline__ void load_group(const void* ptr, long long g, float* f) {
  if (F16) {
    if (PIX == 2) unpack_h8(__ldcs(reinterpret_cast<const uint4*>(ptr) + g), f);
    else unpack_h4(__ldcs(reinterpret_cast<const uint2*>(ptr) + g), f);
  } else {
#pragma unroll
    for (int q = 0; q < PIX; ++q) {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(ptr) + g * PIX + q);
      f[4 * q] = v.x; f[4 * q + 1] = v.y; f[4 * q + 2] = v.z; f[4 * q + 3] = v.w;
    }
  }
}

template <int PIX, bool F16>
__device__ __forceinline__ void fold_range(const LayerTable& lt, int k0, int k1, long long g,
                                           float* acc) {
  int k = k0;
  for (; k + 4 <= k1; k += 4) {
    float v[4][4 * PIX];
#pragma unroll
    for (int j = 0; j < 4; ++j) load_group<PIX, F16>(lt.p[k + j], g, v[j]);
#pragma unroll
    for (int j = 0; j < 4; ++j) fold<PIX>(acc, v[j]);
  }
  for (; k < k1; ++k) {
    float v[4 * PIX];
    load_group<PIX, F16>(lt.p[k], g, v);
    fold<PIX>(acc, v);
  }
}

template <int PIX>
__device__ __forceinline__ void store_group(void* out, int f16, long long g, const float* acc) {
  if (!out) return;
  if (f16) {
    unsigned w[2 * PIX];
#pragma unroll
    for (int k = 0; k < 2 * PIX; ++k) {
      const __half2 h = __floats2half2_rn(acc[2 * k], acc[2 * k + 1]);
      w[k] = *reinterpret_cast<const unsigned*>(&h);
    }
    if (PIX == 2) reinterpret_cast<uint4*>(out)[g] = make_uint4(w[0], w[1], w[2], w[3]);
    else reinterpret_cast<uint2*>(out)[g] = make_uint2(w[0], w[1]);
  } else {
#pragma unroll
    for (int q = 0; q < PIX; ++q)
      reinterpret_cast<float4*>(out)[g * PIX + q] =
          make_float4(acc[4 * q], acc[4 * q + 1], acc[4 * q + 2], acc[4 * q + 3]);
  }
}

template <int PIX, bool F16>
__global__ void __launch_bounds__(256)
composite_kernel(const __grid_constant__ LayerTable lt, int nf, int nb, long long groups,
                 void* Fout, void* Bout, int out_f16) {
  pdl_prologue();
  for (long long g = blockIdx.x * (long long)blockDim.x + threadIdx.x; g < groups;
       g += (long long)gridDim.x * blockDim.x) {
    float acc[4 * PIX];
    if (Fout) {
#pragma unroll
      for (int c = 0; c < 4 * PIX; ++c) acc[c] = 0.f;
      fold_range<PIX, F16>(lt, 0, nf, g, acc);
      store_group<PIX>(Fout, out_f16, g, acc);
    }
    if (Bout) {
#pragma unroll
      for (int c = 0; c < 4 * PIX; ++c) acc[c] = 0.f;
      fold_range<PIX, F16>(lt, nf, nf + nb, g, acc);
      store_group<PIX>(Bout, out_f16, g, acc);
    }
  }
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_composite_cache(abcd_ctx* ctx, const void* const* layers, int L,
                                            int layer_dtype, const int* order, int split,
                                            int width, int height, void* F_out, void* B_out,
                                            int out_dtype) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (L < 0 || L > kMaxLayers || (L > 0 && (!layers || !order)) || split < 0 || split > L ||
      width <= 0 || height <= 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache: bad layer list, split or size");
  if ((layer_dtype != ABCD_F16 && layer_dtype != ABCD_F32) || (out_dtype != ABCD_F16 && out_dtype != ABCD_F32))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache: bad dtype");
  LayerTable lt;
  int nf = 0, nb = 0;
  bool al16 = true;
  for (int k = 0; k < L; ++k) {
    if (k == split) continue;
    if (order[k] < 0 || order[k] >= L) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache: order[%d] out of range", k);
    const void* p = layers[order[k]];
    if (!p) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache: layer %d is NULL", order[k]);
    if ((uintptr_t)p & 15) al16 = false;
    if ((uintptr_t)p & (layer_dtype == ABCD_F16 ? 7 : 15))
      return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache: layer %d misaligned", order[k]);
    if (k < split) lt.p[nf++] = p;
  }
  for (int k = split + 1; k < L; ++k) lt.p[nf + nb++] = layers[order[k]];
  const long long npix = (long long)width * height;
  const uintptr_t oal = out_dtype == ABCD_F16 ? 7 : 15;
  if (((uintptr_t)F_out & oal) || ((uintptr_t)B_out & oal))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache: misaligned output");
  if (((uintptr_t)F_out & 15) || ((uintptr_t)B_out & 15)) al16 = false;
  if (!F_out && !B_out) return ABCD_OK;
  const int grid = ctx->num_sms * 8;
  const bool pairs = al16 && (npix % 2 == 0);
  const bool o16 = out_dtype == ABCD_F16;
  const long long units = pairs ? npix / 2 : npix;
  cudaError_t e;
  if (layer_dtype == ABCD_F16)
    e = pairs ? launch_pdl(composite_kernel<2, true>, dim3(grid), dim3(256), 0, ctx->stream, lt, nf, nb, units, F_out, B_out, o16)
              : launch_pdl(composite_kernel<1, true>, dim3(grid), dim3(256), 0, ctx->stream, lt, nf, nb, units, F_out, B_out, o16);
  else
    e = pairs ? launch_pdl(composite_kernel<2, false>, dim3(grid), dim3(256), 0, ctx->stream, lt, nf, nb, units, F_out, B_out, o16)
              : launch_pdl(composite_kernel<1, false>, dim3(grid), dim3(256), 0, ctx->stream, lt, nf, nb, units, F_out, B_out, o16);
  return check_launch(ctx, "composite_kernel", e);
}

// ---- K1 over packed layers (the cache's tile-sparse format, see abcd_render_refresh_packed):
// one CTA per 16x16 tile, two pixels per thread, the tile's map entries of all layers read
// once into shared memory; a layer whose tile is not stored is
// transparent, and folding (0, 0, 0, 0) leaves the accumulator unchanged, so skipping it gives
// the dense result bit for bit.  Only the stored tiles are read.
namespace abcd {
namespace {

struct PackedTable {
  const int* map[kMaxLayers];       // front layers in order, then back layers in order
  const uint4* data[kMaxLayers];    // 16-byte units: two fp16 RGBA pixels
};

constexpr int kPackedThreads = kTileThreads / 2;

// acc (2 pixels) = acc over the two pixels of every layer in [k0, k1) stored at this tile;
// m: the tile's block index in every layer (shared memory, -1: not stored).  Eight layers'
// loads are in flight before they are folded.
constexpr int kPackedInFlight = 8;

__device__ __forceinline__ void fold_packed(const PackedTable& pt, const int* m, int k0, int k1,
                                            int unit, float* acc) {
  int k = k0;
  for (; k + kPackedInFlight <= k1; k += kPackedInFlight) {
    uint4 r[kPackedInFlight];
#pragma unroll
    for (int j = 0; j < kPackedInFlight; ++j)
      r[j] = m[k + j] >= 0 ? __ldcs(pt.data[k + j] + (size_t)m[k + j] * kPackedThreads + unit)
                           : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int j = 0; j < kPackedInFlight; ++j) {
      if (m[k + j] < 0) continue;
      float v[8];
      unpack_h8(r[j], v);
      fold<2>(acc, v);
    }
  }
  for (; k < k1; ++k) {
    if (m[k] < 0) continue;
    float v[8];
    unpack_h8(__ldcs(pt.data[k] + (size_t)m[k] * kPackedThreads + unit), v);
    fold<2>(acc, v);
  }
}

__device__ __forceinline__ void store_pixel_out(void* out, int f16, long long p, const float* acc) {
  if (f16) {
    const __half2 lo = __floats2half2_rn(acc[0], acc[1]), hi = __floats2half2_rn(acc[2], acc[3]);
    reinterpret_cast<uint2*>(out)[p] = make_uint2(*reinterpret_cast<const unsigned*>(&lo),
                                                  *reinterpret_cast<const unsigned*>(&hi));
  } else {
    reinterpret_cast<float4*>(out)[p] = make_float4(acc[0], acc[1], acc[2], acc[3]);
  }
}

__global__ void __launch_bounds__(kPackedThreads)
composite_packed_kernel(const __grid_constant__ PackedTable pt, int nf, int nb, int width,
                        int height, int tiles_x, void* Fout, void* Bout, int out_f16) {
  pdl_prologue();
  __shared__ int s_map[kMaxLayers];
  const int tile = blockIdx.x;
  const int unit = threadIdx.x;                       // pixels 2 unit, 2 unit + 1 of the tile
  for (int k = threadIdx.x; k < nf + nb; k += blockDim.x) s_map[k] = __ldg(pt.map[k] + tile);
  __syncthreads();
  const int r = unit / (kTile / 2), c = 2 * (unit % (kTile / 2));
  const int y = (tile / tiles_x) * kTile + r, x = (tile % tiles_x) * kTile + c;
  for (int side = 0; side < 2; ++side) {
    void* out = side ? Bout : Fout;
    if (!out) continue;
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
    if (side == 0) fold_packed(pt, s_map, 0, nf, unit, acc);
    else fold_packed(pt, s_map, nf, nf + nb, unit, acc);
    if (y < height) {
      if (x < width) store_pixel_out(out, out_f16, (long long)y * width + x, acc);
      if (x + 1 < width) store_pixel_out(out, out_f16, (long long)y * width + x + 1, acc + 4);
    }
  }
}

}  // namespace
}  // namespace abcd

extern "C" abcd_status abcd_composite_cache_packed(abcd_ctx* ctx, const int* const* tile_maps,
                                                   const void* const* packed, int L,
                                                   const int* order, int split, int width,
                                                   int height, void* F_out, void* B_out,
                                                   int out_dtype) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (L < 0 || L > kMaxLayers || (L > 0 && (!tile_maps || !packed || !order)) || split < 0 ||
      split > L || width <= 0 || height <= 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache_packed: bad layer list, split or size");
  if (out_dtype != ABCD_F16 && out_dtype != ABCD_F32)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache_packed: bad dtype");
  PackedTable pt;
  int nf = 0, nb = 0;
  for (int k = 0; k < L; ++k) {
    if (k == split) continue;
    if (order[k] < 0 || order[k] >= L)
      return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache_packed: order[%d] out of range", k);
    const int* m = tile_maps[order[k]];
    const void* d = packed[order[k]];
    if (!m || !d) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache_packed: layer %d is NULL", order[k]);
    if (((uintptr_t)d & 15) || ((uintptr_t)m & 3))
      return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache_packed: layer %d misaligned", order[k]);
    const int slot = k < split ? nf++ : -1;
    if (slot >= 0) { pt.map[slot] = m; pt.data[slot] = (const uint4*)d; }
  }
  for (int k = split + 1; k < L; ++k) {
    pt.map[nf + nb] = tile_maps[order[k]];
    pt.data[nf + nb] = (const uint4*)packed[order[k]];
    ++nb;
  }
  const uintptr_t oal = out_dtype == ABCD_F16 ? 7 : 15;
  if (((uintptr_t)F_out & oal) || ((uintptr_t)B_out & oal))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_cache_packed: misaligned output");
  if (!F_out && !B_out) return ABCD_OK;
  const int tiles_x = (width + kTile - 1) / kTile, tiles_y = (height + kTile - 1) / kTile;
  return check_launch(ctx, "composite_packed_kernel",
                      launch_pdl(composite_packed_kernel, dim3(tiles_x * tiles_y),
                                 dim3(kPackedThreads), 0, ctx->stream, pt, nf, nb, width, height,
                                 tiles_x, F_out, B_out, out_dtype == ABCD_F16 ? 1 : 0));
}
