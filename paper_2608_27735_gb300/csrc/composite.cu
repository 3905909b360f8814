// K1: depth-ordered over-compositing of cached per-partition RGBA renders into F and B.
// Section 2 builds, per camera, the foreground and background images from the stored renders
// of the frozen partitions in the camera's depth order; by associativity of 'over' the frozen
// blocks in front of the active partition collapse into F, those behind it into B.
//
// Pure streaming work: every layer is read once (16-byte streaming loads, evict-first), the
// accumulator stays in registers across layers, F and B are written once.  Four layers are
// loaded before they are folded so each thread keeps 64 bytes in flight.  The grid is a
// multiple of the SM count and strides over pixel pairs.
#include <algorithm>

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
// once into shared memory; a layer whose tile is not stored is transparent, and folding
// (0, 0, 0, 0) leaves the accumulator unchanged, so skipping it gives the dense result bit for
// bit.  Only the stored tiles are read.
namespace abcd {
namespace {

struct PackedTable {
  const int* map[kMaxLayers];       // front layers in order, then back layers in order
  const uint4* data[kMaxLayers];    // 2 KB blocks of 16-byte units: two fp16 RGBA pixels
};

constexpr int kPackedThreads = kTileThreads / 2;
constexpr int kPackedInFlight = 8;

// The positions k in [0, n) with s_map[k] >= 0, in order, into s_list; returns how many (every
// thread).  Warp 0 compacts with ballots; the caller's next __syncthreads publishes s_list.
__device__ __forceinline__ void compact_stored(const int* s_map, int n, int* s_list,
                                               int* s_count) {
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  int run = 0;
  for (int k0 = 0; k0 < n; k0 += 32) {
    const bool st = k0 + lane < n && s_map[k0 + lane] >= 0;
    const unsigned b = __ballot_sync(0xffffffffu, st);
    if (st) s_list[run + __popc(b & ((1u << lane) - 1u))] = k0 + lane;
    run += __popc(b);
  }
  if (lane == 0) *s_count = run;
}

// Calls fn(k, v) in order for the listed positions s_list[j0 .. j1) (v: this thread's 16-byte
// unit of layer k's block at the tile), the loads of kPackedInFlight blocks in flight before
// they are used.
template <typename Fn>
__device__ __forceinline__ void for_each_listed(const uint4* const* data, const int* s_map,
                                                const int* s_list, int j0, int j1, Fn fn) {
  const int unit = threadIdx.x;
  int j = j0;
  for (; j + kPackedInFlight <= j1; j += kPackedInFlight) {
    uint4 r[kPackedInFlight];
#pragma unroll
    for (int i = 0; i < kPackedInFlight; ++i) {
      const int k = s_list[j + i];
      r[i] = __ldcs(data[k] + (size_t)s_map[k] * kPackedThreads + unit);
    }
#pragma unroll
    for (int i = 0; i < kPackedInFlight; ++i) fn(s_list[j + i], r[i]);
  }
  if (j < j1) {
    uint4 r[kPackedInFlight];
#pragma unroll
    for (int i = 0; i < kPackedInFlight; ++i) {
      if (j + i >= j1) break;
      const int k = s_list[j + i];
      r[i] = __ldcs(data[k] + (size_t)s_map[k] * kPackedThreads + unit);
    }
#pragma unroll
    for (int i = 0; i < kPackedInFlight; ++i) {
      if (j + i >= j1) break;
      fn(s_list[j + i], r[i]);
    }
  }
}

// acc (2 pixels) = acc over the two pixels of every layer in [k0, k1) stored at this tile;
// m: the tile's block index in every layer (shared memory, -1: not stored).  Eight layers'
// loads are in flight before they are folded.
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

// One side's left fold continued from an fp32 accumulator: acc = acc over the listed layers, in
// order (acc_in NULL: from transparent); the accumulator goes back in fp32 (acc_out) and/or as
// its fp16 rounding (out16).  The fold runs the same fp32 operations in the same order as
// composite_packed_kernel, so folding the layers in pieces gives its result bit for bit.
__global__ void __launch_bounds__(kPackedThreads)
fold_packed_kernel(const __grid_constant__ PackedTable pt, int n, int width, int height,
                   int tiles_x, const float4* acc_in, float4* acc_out, uint2* out16) {
  pdl_prologue();
  __shared__ int s_map[kMaxLayers];
  const int tile = blockIdx.x;
  const int unit = threadIdx.x;
  for (int k = threadIdx.x; k < n; k += blockDim.x) s_map[k] = __ldg(pt.map[k] + tile);
  __syncthreads();
  const int r = unit / (kTile / 2), c = 2 * (unit % (kTile / 2));
  const int y = (tile / tiles_x) * kTile + r, x = (tile % tiles_x) * kTile + c;
  const long long p0 = (long long)y * width + x;
  const bool in0 = y < height && x < width, in1 = y < height && x + 1 < width;
  float acc[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) acc[q] = 0.f;
  if (acc_in) {
    if (in0) { const float4 a = acc_in[p0]; acc[0] = a.x; acc[1] = a.y; acc[2] = a.z; acc[3] = a.w; }
    if (in1) { const float4 a = acc_in[p0 + 1]; acc[4] = a.x; acc[5] = a.y; acc[6] = a.z; acc[7] = a.w; }
  }
  fold_packed(pt, s_map, 0, n, unit, acc);
  if (in0) {
    if (acc_out) acc_out[p0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    if (out16) store_pixel_out(out16, 1, p0, acc);
  }
  if (in1) {
    if (acc_out) acc_out[p0 + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    if (out16) store_pixel_out(out16, 1, p0 + 1, acc + 4);
  }
}

}  // namespace
}  // namespace abcd

extern "C" abcd_status abcd_composite_fold_packed(abcd_ctx* ctx, const int* const* tile_maps,
                                                  const void* const* packed, int count,
                                                  int width, int height, const float* acc_in,
                                                  float* acc_out, void* out16) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (count < 0 || count > kMaxLayers || (count > 0 && (!tile_maps || !packed)) || width <= 0 ||
      height <= 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_fold_packed: bad layer list or size");
  if (((uintptr_t)acc_in & 15) || ((uintptr_t)acc_out & 15) || ((uintptr_t)out16 & 7))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_fold_packed: misaligned accumulator or output");
  PackedTable pt;
  for (int k = 0; k < count; ++k) {
    const int* m = tile_maps[k];
    const void* d = packed[k];
    if (!m || !d) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_fold_packed: layer %d is NULL", k);
    if (((uintptr_t)d & 15) || ((uintptr_t)m & 3))
      return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_composite_fold_packed: layer %d misaligned", k);
    pt.map[k] = m;
    pt.data[k] = (const uint4*)d;
  }
  if (!acc_out && !out16) return ABCD_OK;
  const int tiles_x = (width + kTile - 1) / kTile, tiles_y = (height + kTile - 1) / kTile;
  return check_launch(ctx, "fold_packed_kernel",
                      launch_pdl(fold_packed_kernel, dim3(tiles_x * tiles_y), dim3(kPackedThreads),
                                 0, ctx->stream, pt, count, width, height, tiles_x,
                                 (const float4*)acc_in, (float4*)acc_out, (uint2*)out16));
}

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

// ---- visibility of the layers of one camera's depth order (Section 4: visibility thresholds
// and occlusion culling of camera-partition pairs).  For the layer at position k, with alpha_k
// its alpha and T_k the product of (1 - alpha) over the layers before it, visible = mean over
// pixels of alpha_k T_k and coverage = mean of alpha_k.  Leaving a set D of layers out of the
// composite changes every channel of every pixel by at most the sum over D of alpha_j T_j
// (colours premultiplied and at most alpha), so the dropped layers' visible shares bound the
// mean error of a culled composite.
// One CTA per 16x16 tile at a time (a grid that strides over tiles), two pixels per thread, T
// in registers across the order.  Sums are exact: every value is rounded to 24-bit fixed point
// and added as an integer (a warp reduction, then 64-bit shared and global accumulators), so
// the result does not depend on the order of the additions; CTAs add to one of kVisCopies
// copies of the global sums (fewer atomics on one address) and the last CTA to finish adds the
// copies, converts them to means and clears them for the next call.
namespace abcd {
namespace {

constexpr float kVisScale = 16777216.f;       // 2^24
constexpr int kVisInFlight = 8;               // layers whose loads are in flight together
constexpr int kVisCopies = kVisSumCopies;     // global accumulators (CTA b adds to copy b % 8)

struct VisTable {
  const int* map[kMaxLayers];                 // packed: tile map per position of the order
  const uint4* data[kMaxLayers];              // packed: 2 KB blocks; dense: half [H][W][4]
  int layer[kMaxLayers];                      // layer index at each position
};

// Adds one layer's contribution at the thread's two pixels (alphas a0, a1) to the CTA's sums
// of position k, then takes the layer's transmittance factor into T0, T1.  Warp-uniform k.
__device__ __forceinline__ void vis_accumulate(float a0, float a1, float& T0, float& T1, int k,
                                               unsigned long long (*s_sum)[kMaxLayers]) {
  const unsigned vf = __float2uint_rn(a0 * T0 * kVisScale) + __float2uint_rn(a1 * T1 * kVisScale);
  const unsigned cf = __float2uint_rn(a0 * kVisScale) + __float2uint_rn(a1 * kVisScale);
  T0 *= 1.f - a0;
  T1 *= 1.f - a1;
  const unsigned vs = __reduce_add_sync(0xffffffffu, vf);
  const unsigned cs = __reduce_add_sync(0xffffffffu, cf);
  if ((threadIdx.x & 31) == 0) {
    if (vs) atomicAdd(&s_sum[0][k], (unsigned long long)vs);
    if (cs) atomicAdd(&s_sum[1][k], (unsigned long long)cs);
  }
}

__device__ __forceinline__ float alpha_hi(unsigned w) {
  return __high2float(*reinterpret_cast<const __half2*>(&w));
}

template <bool PACKED>
__global__ void __launch_bounds__(kPackedThreads, 10)
visibility_kernel(const __grid_constant__ VisTable vt, int count, int L, int width, int height,
                  int tiles_x, int n_tiles, unsigned long long* sums, unsigned* ticket,
                  double* visible, double* coverage) {
  pdl_prologue();
  __shared__ unsigned long long s_sum[2][kMaxLayers];
  __shared__ int s_map[kMaxLayers];
  __shared__ int s_list[kMaxLayers];
  __shared__ int s_count;
  __shared__ bool s_last;
  for (int k = threadIdx.x; k < count; k += blockDim.x) { s_sum[0][k] = 0ull; s_sum[1][k] = 0ull; }
  const int unit = threadIdx.x;
  const int r = unit / (kTile / 2), c = 2 * (unit % (kTile / 2));
  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    __syncthreads();                                   // s_map, s_list of the previous tile done
    if (PACKED) {
      for (int k = threadIdx.x; k < count; k += blockDim.x) s_map[k] = __ldg(vt.map[k] + tile);
      __syncthreads();
      compact_stored(s_map, count, s_list, &s_count);
    }
    __syncthreads();
    const int y = (tile / tiles_x) * kTile + r, x = (tile % tiles_x) * kTile + c;
    const bool in0 = y < height && x < width, in1 = y < height && x + 1 < width;
    float T0 = 1.f, T1 = 1.f;
    if (PACKED) {
      for_each_listed(vt.data, s_map, s_list, 0, s_count, [&](int k, uint4 u) {
        vis_accumulate(in0 ? alpha_hi(u.y) : 0.f, in1 ? alpha_hi(u.w) : 0.f, T0, T1, k, s_sum);
      });
      continue;
    }
    const long long p = (long long)y * width + x;
    for (int k0 = 0; k0 < count; k0 += kVisInFlight) {
      // the loads of kVisInFlight layers are issued before any is used (they do not depend on
      // T), so a tile waits for memory once per group instead of once per layer
      unsigned w0[kVisInFlight], w1[kVisInFlight];
#pragma unroll
      for (int j = 0; j < kVisInFlight; ++j) {
        w0[j] = w1[j] = 0u;
        const int k = k0 + j;
        if (k >= count) continue;
        const uint2* d = reinterpret_cast<const uint2*>(vt.data[k]);
        if (in0) w0[j] = __ldcs(d + p).y;
        if (in1) w1[j] = __ldcs(d + p + 1).y;
      }
#pragma unroll
      for (int j = 0; j < kVisInFlight; ++j)
        if (k0 + j < count)
          vis_accumulate(alpha_hi(w0[j]), alpha_hi(w1[j]), T0, T1, k0 + j, s_sum);
    }
  }
  __syncthreads();
  unsigned long long* mine = sums + (size_t)(blockIdx.x % kVisCopies) * 2 * kMaxLayers;
  for (int k = threadIdx.x; k < count; k += blockDim.x) {
    if (s_sum[0][k]) atomicAdd(mine + k, s_sum[0][k]);
    if (s_sum[1][k]) atomicAdd(mine + kMaxLayers + k, s_sum[1][k]);
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const double inv = 1.0 / ((double)kVisScale * (double)width * (double)height);
  for (int j = threadIdx.x; j < L; j += blockDim.x) {
    visible[j] = 0.0;
    if (coverage) coverage[j] = 0.0;
  }
  __syncthreads();
  for (int k = threadIdx.x; k < count; k += blockDim.x) {
    unsigned long long v = 0ull, cv = 0ull;
    for (int cp = 0; cp < kVisCopies; ++cp) {
      v += atomicExch(sums + (size_t)cp * 2 * kMaxLayers + k, 0ull);
      cv += atomicExch(sums + (size_t)cp * 2 * kMaxLayers + kMaxLayers + k, 0ull);
    }
    visible[vt.layer[k]] = (double)v * inv;
    if (coverage) coverage[vt.layer[k]] = (double)cv * inv;
  }
  if (threadIdx.x == 0) *ticket = 0u;
}

// Checks the order and the outputs, fills vt.layer and launches.
abcd_status visibility_launch(abcd_ctx* ctx, const char* who, VisTable& vt, bool packed, int L,
                              const int* order, int count, int width, int height,
                              double* visible, double* coverage) {
  if (!visible || ((uintptr_t)visible & 7) || ((uintptr_t)coverage & 7))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "%s: null or misaligned output", who);
  const int tiles_x = (width + kTile - 1) / kTile, tiles_y = (height + kTile - 1) / kTile;
  const int n_tiles = tiles_x * tiles_y;
  const int grid = std::max(1, std::min(n_tiles, 8 * ctx->num_sms));
  const auto kernel = packed ? visibility_kernel<true> : visibility_kernel<false>;
  return check_launch(ctx, "visibility_kernel",
                      launch_pdl(kernel, dim3(grid), dim3(kPackedThreads), 0, ctx->stream, vt,
                                 count, L, width, height, tiles_x, n_tiles, ctx->ws.vis_sums,
                                 ctx->ws.vis_ticket, visible, coverage));
}

// The order: count distinct indices below L.
bool valid_order(const int* order, int count, int L) {
  unsigned char seen[kMaxLayers] = {0};
  for (int k = 0; k < count; ++k) {
    if (order[k] < 0 || order[k] >= L || seen[order[k]]) return false;
    seen[order[k]] = 1;
  }
  return true;
}

}  // namespace
}  // namespace abcd

extern "C" abcd_status abcd_layer_visibility(abcd_ctx* ctx, const void* const* layers, int L,
                                             const int* order, int count, int width, int height,
                                             double* visible, double* coverage) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_layer_visibility: no workspace");
  if (L < 0 || L > kMaxLayers || count < 0 || count > L || (count > 0 && (!layers || !order)) ||
      width <= 0 || height <= 0 || !valid_order(order, count, L))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_layer_visibility: bad layer list, order or size");
  VisTable vt;
  for (int k = 0; k < count; ++k) {
    const void* p = layers[order[k]];
    if (!p || ((uintptr_t)p & 7))
      return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_layer_visibility: layer %d is NULL or misaligned", order[k]);
    vt.map[k] = nullptr;
    vt.data[k] = static_cast<const uint4*>(p);
    vt.layer[k] = order[k];
  }
  return visibility_launch(ctx, "abcd_layer_visibility", vt, false, L, order, count, width,
                           height, visible, coverage);
}

extern "C" abcd_status abcd_layer_visibility_packed(abcd_ctx* ctx, const int* const* tile_maps,
                                                    const void* const* packed, int L,
                                                    const int* order, int count, int width,
                                                    int height, double* visible,
                                                    double* coverage) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_layer_visibility_packed: no workspace");
  if (L < 0 || L > kMaxLayers || count < 0 || count > L ||
      (count > 0 && (!tile_maps || !packed || !order)) || width <= 0 || height <= 0 ||
      !valid_order(order, count, L))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_layer_visibility_packed: bad layer list, order or size");
  VisTable vt;
  for (int k = 0; k < count; ++k) {
    const int* m = tile_maps[order[k]];
    const void* d = packed[order[k]];
    if (!m || !d || ((uintptr_t)d & 15) || ((uintptr_t)m & 3))
      return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_layer_visibility_packed: layer %d is NULL or misaligned", order[k]);
    vt.map[k] = m;
    vt.data[k] = static_cast<const uint4*>(d);
    vt.layer[k] = order[k];
  }
  return visibility_launch(ctx, "abcd_layer_visibility_packed", vt, true, L, order, count,
                           width, height, visible, coverage);
}
