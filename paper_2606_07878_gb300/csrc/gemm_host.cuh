// Host side of the tcgen05 GEMM: TMA descriptors, tile/split bookkeeping, launch.
#pragma once
#include <algorithm>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstring>
#include <mutex>

#include "epilogues.cuh"

namespace still {

// A 2-D row-major 16-bit operand as TMA sees it: `rows` rows of `cols` elements, row pitch
// `pitch` elements (pitch * 2 must be a multiple of 16 and ptr 16-byte aligned).
struct Operand2D {
  const void* ptr = nullptr;
  int64_t rows = 0, cols = 0, pitch = 0;
};

inline PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// A 3-D destination for TMA stores: element (x, y, z) at base + z * zstride + y * ystride + x
// (elements), extents (nx, ny, nz); boxes of bx x 32 x 1, optionally 128-byte swizzled.
struct StoreView3D {
  void* ptr = nullptr;
  int elem_bytes = 2;
  int64_t nx = 0, ny = 0, nz = 1, ystride = 0, zstride = 0;
  int bx = 32;
  bool swizzle128 = false;
};

inline bool make_store_tmap(CUtensorMap* m, const StoreView3D& v) {
  auto enc = tensor_map_encoder();
  if (enc == nullptr) return false;
  const int64_t eb = v.elem_bytes;
  if ((reinterpret_cast<uintptr_t>(v.ptr) & 15) != 0 || (v.ystride * eb) % 16 != 0 ||
      (v.zstride * eb) % 16 != 0 || (v.bx * eb) % 16 != 0)
    return false;
  cuuint64_t dims[3] = {(cuuint64_t)v.nx, (cuuint64_t)v.ny, (cuuint64_t)v.nz};
  cuuint64_t strides[2] = {(cuuint64_t)(v.ystride * eb), (cuuint64_t)(v.zstride * eb)};
  cuuint32_t box[3] = {(cuuint32_t)v.bx, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, eb == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                   3, v.ptr, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   v.swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                   CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Box = box_rows x 64 elements, 128-byte swizzle, zero fill out of bounds.
inline bool make_tmap(CUtensorMap* m, const Operand2D& op, int box_rows) {
  auto enc = tensor_map_encoder();
  if (enc == nullptr) return false;
  if ((reinterpret_cast<uintptr_t>(op.ptr) & 15) != 0 || (op.pitch * 2) % 16 != 0) return false;
  cuuint64_t dims[2] = {(cuuint64_t)op.cols, (cuuint64_t)op.rows};
  cuuint64_t strides[1] = {(cuuint64_t)(op.pitch * 2)};
  cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(op.ptr), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Fills the derived fields of p. Returns false on an invalid description.
template <int BN>
inline bool finalize_gemm(GemmParams& p, int ab_fmt) {
  if (p.M <= 0 || p.N <= 0 || p.batch <= 0 || p.npass < 1 || p.npass > 3 || p.bdiv < 1)
    return false;
  int iters = 0;
  for (int i = 0; i < p.npass; ++i) {
    if (p.pass[i].klen <= 0 || p.pass[i].klen % kBK != 0) return false;
    if (p.pass[i].a_koff % 8 != 0 || p.pass[i].b_koff % 8 != 0) return false;
    iters += p.pass[i].klen / kBK;
  }
  if ((p.a_k0 | p.a_k1 | p.b_k0 | p.b_k1) % 8 != 0) return false;
  p.iters_total = iters;
  if (p.ksplit < 1) p.ksplit = 1;
  if (p.ksplit > iters) p.ksplit = iters;
  p.tiles_m = (p.M + kBM - 1) / kBM;
  p.tiles_n = (p.N + BN - 1) / BN;
  const int64_t nt = (int64_t)p.tiles_m * p.tiles_n * p.ksplit * p.batch;
  if (nt > 0x7fffffff) return false;
  p.ntiles = (int)nt;
  p.idesc = idesc_f16(kBM, BN, ab_fmt);
  return true;
}

template <int BN, int kRole, class Epi>
inline cudaError_t launch_gemm(const Operand2D& A, const Operand2D& B, GemmParams p, Epi epi,
                               int ab_fmt, int num_sms, cudaStream_t stream,
                               const StoreView3D* out_view = nullptr) {
  using S = GemmSmem<BN, Epi>;
  if (!finalize_gemm<BN>(p, ab_fmt)) return cudaErrorInvalidValue;
  CUtensorMap ta, tb, tc;
  if (!make_tmap(&ta, A, kBM) || !make_tmap(&tb, B, BN)) return cudaErrorInvalidValue;
  std::memset(&tc, 0, sizeof(tc));
  if (out_view != nullptr && !make_store_tmap(&tc, *out_view)) return cudaErrorInvalidValue;
  epi.tile_cols_ = BN;
  auto kern = tc_gemm_kernel<BN, Epi, kRole>;
  static thread_local bool attr_set = false;  // per instantiation
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int grid = p.ntiles < num_sms ? p.ntiles : num_sms;
  kern<<<grid, gemm_threads<Epi>(), S::kBytes, stream>>>(ta, tb, tc, p, epi);
  return cudaGetLastError();
}

// The 2-SM form (tc_gemm2_kernel) on clusters of two CTAs: one 256 x BN tile per pair.
template <int BN, int kRole, class Epi>
inline cudaError_t launch_gemm_2sm(const Operand2D& A, const Operand2D& B, GemmParams p, Epi epi,
                                   int ab_fmt, int num_sms, cudaStream_t stream,
                                   const StoreView3D* out_view = nullptr) {
  using S = Gemm2Smem<BN, Epi>;
  if (!finalize_gemm<BN>(p, ab_fmt)) return cudaErrorInvalidValue;
  CUtensorMap ta, tb, tc;
  if (!make_tmap(&ta, A, kBM) || !make_tmap(&tb, B, BN / 2)) return cudaErrorInvalidValue;
  std::memset(&tc, 0, sizeof(tc));
  if (out_view != nullptr && !make_store_tmap(&tc, *out_view)) return cudaErrorInvalidValue;
  epi.tile_cols_ = BN;
  auto kern = tc_gemm2_kernel<BN, Epi, kRole>;
  static thread_local int clusters = 0;  // per instantiation: resident clusters of two
  if (clusters == 0) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kBytes);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t q = {};
    q.gridDim = dim3(2 * std::max(1, num_sms / 2), 1, 1);
    q.blockDim = dim3(gemm_threads<Epi>(), 1, 1);
    q.dynamicSmemBytes = S::kBytes;
    cudaLaunchAttribute qa[1];
    qa[0].id = cudaLaunchAttributeClusterDimension;
    qa[0].val.clusterDim.x = 2;
    qa[0].val.clusterDim.y = 1;
    qa[0].val.clusterDim.z = 1;
    q.attrs = qa;
    q.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &q) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    clusters = std::max(1, std::min(n, num_sms / 2));
  }
  const int64_t npairs = (int64_t)((p.tiles_m + 1) / 2) * p.tiles_n * p.ksplit * p.batch;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(gemm_threads<Epi>(), 1, 1);
  cfg.dynamicSmemBytes = S::kBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(2 * (unsigned)std::min<int64_t>(npairs, clusters), 1, 1);
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, p, epi);
}

}  // namespace still
