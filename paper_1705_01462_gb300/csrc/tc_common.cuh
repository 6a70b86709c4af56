// Helpers shared by the tensor-core contraction kernels (device: operand layouts and
// conversions; host: TMA tensor maps).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdint>
#include <mutex>

#include "fgq_device.cuh"
#include "ptx_sm100.cuh"

namespace fgq {
namespace tc {

// Byte offset of 16-byte chunk c (0..7) of row r in a 128B-swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128(int r, int c) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

// Byte offset of 16-byte chunk c of staging row t.  Rows are 64 bytes (8-bit activations,
// 4 chunks) or 32 bytes (4-bit, 2 chunks); the chunk index is XOR-ed with row bits so that
// eight consecutive rows read the same chunk from eight different bank groups.  This is
// the layout a TMA box load with the 64-byte (32-byte) swizzle produces.
template <int ABITS>
__device__ __forceinline__ uint32_t st_off(int t, int c) {
  if (ABITS == 8) return (uint32_t)(t * 64 + ((c ^ ((t >> 1) & 3)) << 4));
  return (uint32_t)(t * 32 + ((c ^ ((t >> 2) & 1)) << 4));
}

// fp16 pair (lo, hi) from two 8-bit lanes of x selected by sel (unsigned: 1024 + v - 1024).
__device__ __forceinline__ uint32_t u8pair_to_h2(uint32_t x, uint32_t sel, uint32_t bias2) {
  const uint32_t h = __byte_perm(x, 0x64646464u, sel);  // halves 1024 + v
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(h), "r"(bias2));
  return r;
}

// Expansion of 2-bit codes: a nibble (two codes) -> two fp16 {0, +1, -1}, stored 32 times
// ([16][32] words) so that lane l reads copy l and no two lanes share a bank.
__device__ __forceinline__ void fill_code_lut(uint32_t* lut) {
  for (int i = threadIdx.x; i < 16 * 32; i += blockDim.x) {
    const uint32_t x = (uint32_t)i >> 5;
    uint32_t h[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const uint32_t c = (x >> (2 * e)) & 3u;
      h[e] = c == 1u ? 0x3C00u : (c == 3u ? 0xBC00u : 0u);
    }
    lut[i] = h[0] | (h[1] << 16);
  }
}

// Converts the 64 codes (16 bytes) of one K-tile row to fp16 into row t of a 128B-swizzled
// K-major operand tile; lut = the table above, offset by the calling lane.
__device__ __forceinline__ void codes_row_to_fp16(const uint8_t* codes16, uint8_t* tile, int t, const uint32_t* lt) {
  uint32_t cw[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) cw[i] = *reinterpret_cast<const uint32_t*>(codes16 + 4 * i);
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const uint32_t bits = (cw[c / 2] >> (16 * (c & 1))) & 0xffffu;  // 8 codes
    *reinterpret_cast<uint4*>(tile + sw128(t, c)) =
        make_uint4(lt[32 * (bits & 15u)], lt[32 * ((bits >> 4) & 15u)], lt[32 * ((bits >> 8) & 15u)], lt[32 * (bits >> 12)]);
  }
}

// Half h (codes 32 h .. 32 h + 31, 8 bytes) of one K-tile row: 16-byte chunks 4 h .. 4 h + 3
// of row t of the 128B-swizzled operand tile.
__device__ __forceinline__ void codes_half_row_to_fp16(const uint8_t* codes16, int h, uint8_t* tile, int t,
                                                       const uint32_t* lt) {
  const uint2 cw = *reinterpret_cast<const uint2*>(codes16 + 8 * h);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t bits = ((i < 2 ? cw.x : cw.y) >> (16 * (i & 1))) & 0xffffu;  // 8 codes
    *reinterpret_cast<uint4*>(tile + sw128(t, 4 * h + i)) =
        make_uint4(lt[32 * (bits & 15u)], lt[32 * ((bits >> 4) & 15u)], lt[32 * ((bits >> 8) & 15u)], lt[32 * (bits >> 12)]);
  }
}

// Raises a kernel's dynamic shared-memory limit to `bytes`, once per device (the attribute
// belongs to the device's context); thread-safe.  Returns false if the call failed.
template <auto Kernel>
bool smem_attr_once(int bytes) {
  constexpr int kDev = 64;
  static std::once_flag once[kDev];
  static bool ok[kDev];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kDev) return false;
  std::call_once(once[dev], [&] {
    ok[dev] = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) == cudaSuccess;
  });
  return ok[dev];
}

// cuTensorMapEncodeTiled from the driver, looked up once through the runtime.
inline PFN_cuTensorMapEncodeTiled_v12000 encode_tiled() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// cuTensorMapEncodeIm2col from the driver, looked up once through the runtime.
inline PFN_cuTensorMapEncodeIm2col_v12000 encode_im2col() {
  static PFN_cuTensorMapEncodeIm2col_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeIm2col_v12000>(p);
  });
  return fn;
}

// im2col map of an NHWC tensor [B][H][W][C] (elements of elem_bytes bytes) for a
// convolution with an R x S filter, stride and zero padding pad: the bounding box of the
// filter windows' top-left pixels runs from -pad to W + pad - S (H + pad - R), walked with
// the convolution's stride, so that consecutive pixels of a column are consecutive output
// positions; each pixel contributes `pixel_elems` channels to a row of the box.
inline bool make_map_im2col(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t C, uint64_t elem_bytes,
                            int B, int H, int W, int R, int S, int stride, int pad, uint32_t pixel_elems,
                            uint32_t pixels, CUtensorMapSwizzle sw) {
  auto enc = encode_im2col();
  if (!enc) return false;
  const uint64_t row = C * elem_bytes;
  const cuuint64_t dims[4] = {C, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)B};
  const cuuint64_t strides[3] = {row, row * (cuuint64_t)W, row * (cuuint64_t)W * (cuuint64_t)H};
  const int lower[2] = {-pad, -pad};                   // {W, H}
  const int upper[2] = {pad - (S - 1), pad - (R - 1)};  // {W, H}
  const cuuint32_t estr[4] = {1, (cuuint32_t)stride, (cuuint32_t)stride, 1};
  return enc(m, dt, 4, const_cast<void*>(base), dims, strides, lower, upper, pixel_elems, pixels, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Whether a convolution's geometry fits an im2col map (the corner offsets of a 4D map are
// 8-bit signed, the traversal stride at most 8).
inline bool im2col_fits(int R, int S, int stride, int pad) {
  const int lo = -pad, up_w = pad - (S - 1), up_h = pad - (R - 1);
  return stride >= 1 && stride <= 8 && lo >= -128 && up_w >= -128 && up_w <= 127 && up_h >= -128 && up_h <= 127;
}

// 2D tiled map: dims {d0 (innermost), d1}, row pitch in bytes, box {b0, b1}.
inline bool make_map_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t d0, uint64_t d1,
                 uint64_t pitch, uint32_t b0, uint32_t b1, CUtensorMapSwizzle sw) {
  auto enc = encode_tiled();
  if (!enc) return false;
  const cuuint64_t dims[2] = {d0, d1};
  const cuuint64_t strides[1] = {pitch};
  const cuuint32_t box[2] = {b0, b1};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
             CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The activations of the tensor-core kernels as fp16 integers (defined with the G >= 64
// kernel): NHWC, or [P][C] -- only the pixels a strided 1x1 unpadded convolution reads.
bool act_pointwise(const Geom& g);         // 1x1, unpadded (any stride), or a GEMM: 2D rows
int64_t act16_elems(const Geom& g);        // elements of the fp16 copy
// 2D map (pointwise) or im2col map of the fp16 copy: boxes of `pixels` output positions x 64
// channels, 128-byte swizzle
bool act16_map(CUtensorMap* m, const void* x16, const Geom& g, uint32_t pixels);
bool act16_supported(const Geom& g);       // C % 16 == 0, Cg % 64 == 0, a map for the geometry

}  // namespace tc
}  // namespace fgq
