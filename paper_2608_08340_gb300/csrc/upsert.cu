// Op_upsert (Sec. 3.2, I' = Op_upsert(I, E; b_u); Sec. 4.1 Upsert): a batch
// of embeddings overwrites rows of the index in one bulk, coalesced pass.
// Duplicate ids are resolved on the host before launch (the later entry of
// the batch wins), so every destination row is written by exactly one warp.
#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

constexpr int kWarpsPerBlock = 8;

// Same element type: one warp copies one row with 16-byte vectors.
__global__ void copy_rows_kernel(uint4* __restrict__ E, int vec_per_row,
                                 const uint4* __restrict__ rows, const int64_t* __restrict__ pairs,
                                 int64_t count) {
  const int64_t w = static_cast<int64_t>(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (w >= count) return;
  const int lane = threadIdx.x & 31;
  const int64_t src = pairs[2 * w], dst = pairs[2 * w + 1];
  for (int v = lane; v < vec_per_row; v += 32)
    E[dst * vec_per_row + v] = rows[src * vec_per_row + v];
}

// fp32 rows into a bf16 index: round to nearest even, 8 values per 16-byte store.
__global__ void convert_rows_kernel(uint4* __restrict__ E, int d, const float4* __restrict__ rows,
                                    const int64_t* __restrict__ pairs, int64_t count) {
  const int64_t w = static_cast<int64_t>(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (w >= count) return;
  const int lane = threadIdx.x & 31;
  const int64_t src = pairs[2 * w], dst = pairs[2 * w + 1];
  const int groups = d / 8;
  for (int v = lane; v < groups; v += 32) {
    const float4 a = rows[(src * d) / 4 + 2 * v];
    const float4 b = rows[(src * d) / 4 + 2 * v + 1];
    __nv_bfloat162 p0 = __floats2bfloat162_rn(a.x, a.y);
    __nv_bfloat162 p1 = __floats2bfloat162_rn(a.z, a.w);
    __nv_bfloat162 p2 = __floats2bfloat162_rn(b.x, b.y);
    __nv_bfloat162 p3 = __floats2bfloat162_rn(b.z, b.w);
    uint4 o;
    o.x = *reinterpret_cast<uint32_t*>(&p0);
    o.y = *reinterpret_cast<uint32_t*>(&p1);
    o.z = *reinterpret_cast<uint32_t*>(&p2);
    o.w = *reinterpret_cast<uint32_t*>(&p3);
    E[(dst * d) / 8 + v] = o;
  }
}

__global__ void convert_kernel(const float4* __restrict__ src, uint2* __restrict__ dst,
                               int64_t count4) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const float4 a = src[i];
    __nv_bfloat162 p0 = __floats2bfloat162_rn(a.x, a.y);
    __nv_bfloat162 p1 = __floats2bfloat162_rn(a.z, a.w);
    uint2 o;
    o.x = *reinterpret_cast<uint32_t*>(&p0);
    o.y = *reinterpret_cast<uint32_t*>(&p1);
    dst[i] = o;
  }
}

}  // namespace

cudaError_t launch_scatter_rows(int index_dtype, void* E, int d, const void* rows, int rows_dtype,
                                const int64_t* pairs, int64_t count, cudaStream_t st) {
  if (count <= 0) return cudaSuccess;
  const unsigned blocks = static_cast<unsigned>((count + kWarpsPerBlock - 1) / kWarpsPerBlock);
  if (index_dtype == rows_dtype) {
    const int elem = index_dtype == kF32 ? 4 : 2;
    copy_rows_kernel<<<blocks, kWarpsPerBlock * 32, 0, st>>>(
        static_cast<uint4*>(E), d * elem / 16, static_cast<const uint4*>(rows), pairs, count);
  } else {
    convert_rows_kernel<<<blocks, kWarpsPerBlock * 32, 0, st>>>(
        static_cast<uint4*>(E), d, static_cast<const float4*>(rows), pairs, count);
  }
  return cudaGetLastError();
}

cudaError_t launch_convert_f32_bf16(const float* src, void* dst, int64_t count, cudaStream_t st) {
  const int64_t count4 = count / 4;
  if (count4 <= 0) return cudaSuccess;
  int64_t blocks = (count4 + 255) / 256;
  if (blocks > 65535) blocks = 65535;
  convert_kernel<<<static_cast<unsigned>(blocks), 256, 0, st>>>(
      reinterpret_cast<const float4*>(src), static_cast<uint2*>(dst), count4);
  return cudaGetLastError();
}

}  // namespace oprag
