// Tail of Op_embed (Sec. 4.3): the hidden states of each chunk or query of a
// padded batch are mean-pooled over its unmasked tokens and L2-normalised,
// and the vector is written in the index's dtype, ready for oprag_search.
//
// One CTA of 256 threads per batch row.  Thread i accumulates, in fp32, the
// 16-byte groups i, i + 256, ... of the row's dim elements over the tokens,
// the loads of kTokenBatch tokens in flight at once (a batch has few rows, so
// each CTA must keep many bytes in flight); a block reduction of the squared
// mean gives the norm.  HBM-bound: the unmasked hidden states are read once.
#include <cuda_bf16.h>

#include "common.cuh"
#include "internal.h"

namespace oprag {

namespace {

constexpr int kPoolThreads = 256;
constexpr int kTokenBatch = 8;

template <typename TIn>
struct Group;                                   // one 16-byte group of inputs
template <>
struct Group<uint16_t> {
  static constexpr int kN = 8;
  __device__ static void add(const uint4& v, float (&a)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      a[2 * i] += __uint_as_float(w[i] << 16);
      a[2 * i + 1] += __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
};
template <>
struct Group<float> {
  static constexpr int kN = 4;
  __device__ static void add(const uint4& v, float (&a)[4]) {
    a[0] += __uint_as_float(v.x);
    a[1] += __uint_as_float(v.y);
    a[2] += __uint_as_float(v.z);
    a[3] += __uint_as_float(v.w);
  }
};

template <typename TIn, int R>
__global__ void __launch_bounds__(kPoolThreads)
embed_pool_kernel(const TIn* __restrict__ hidden, int tokens, int dim,
                  const uint8_t* __restrict__ mask, void* __restrict__ out, int out_bf16) {
  constexpr int N = Group<TIn>::kN;
  __shared__ float red[kPoolThreads / 32];
  __shared__ float total;
  const int b = blockIdx.x;
  const int groups = dim / N;
  const uint4* row0 = reinterpret_cast<const uint4*>(hidden + static_cast<int64_t>(b) * tokens * dim);
  const uint8_t* mrow = mask + static_cast<int64_t>(b) * tokens;
  float acc[R][N];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int i = 0; i < N; ++i) acc[r][i] = 0.f;
  // Tokens are added in increasing order (a fixed summation order).
  constexpr int TB = R <= 2 ? kTokenBatch : kTokenBatch / 2;   // register budget
  int count = 0;
  for (int t = 0; t < tokens; t += TB) {
    bool m[TB];
#pragma unroll
    for (int u = 0; u < TB; ++u) {
      m[u] = t + u < tokens && mrow[t + u] != 0;
      count += static_cast<int>(m[u]);
    }
    uint4 v[TB][R];
#pragma unroll
    for (int u = 0; u < TB; ++u)
#pragma unroll
      for (int r = 0; r < R; ++r) {
        const int g = threadIdx.x + r * kPoolThreads;
        v[u][r] = m[u] && g < groups ? __ldg(row0 + static_cast<int64_t>(t + u) * groups + g)
                                     : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
    for (int u = 0; u < TB; ++u)
#pragma unroll
      for (int r = 0; r < R; ++r)
        if (m[u]) Group<TIn>::add(v[u][r], acc[r]);
  }
  // Mean, then the block-wide sum of its squares.
  const float inv_c = count > 0 ? 1.f / static_cast<float>(count) : 0.f;
  float ss = 0.f;
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int i = 0; i < N; ++i) {
      acc[r][i] *= inv_c;
      ss = fmaf(acc[r][i], acc[r][i], ss);
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int w = 0; w < kPoolThreads / 32; ++w) s += red[w];
    total = s;
  }
  __syncthreads();
  const float norm = sqrtf(total);
  const float scale = count > 0 && norm > 0.f ? 1.f / norm : 0.f;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int g = threadIdx.x + r * kPoolThreads;
    if (g >= groups) continue;
    const int64_t e0 = static_cast<int64_t>(b) * dim + static_cast<int64_t>(g) * N;
    if (out_bf16) {
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(out) + e0;
#pragma unroll
      for (int i = 0; i < N; i += 2)
        *reinterpret_cast<__nv_bfloat162*>(o + i) =
            __floats2bfloat162_rn(acc[r][i] * scale, acc[r][i + 1] * scale);
    } else {
      float* o = static_cast<float*>(out) + e0;
#pragma unroll
      for (int i = 0; i < N; i += 4)
        *reinterpret_cast<float4*>(o + i) = make_float4(acc[r][i] * scale, acc[r][i + 1] * scale,
                                                        acc[r][i + 2] * scale, acc[r][i + 3] * scale);
    }
  }
}

template <typename TIn>
cudaError_t launch_typed(const void* hidden, int batch, int tokens, int dim, const uint8_t* mask,
                         void* out, int out_bf16, cudaStream_t st) {
  const int groups = dim / Group<TIn>::kN;
  const int r = (groups + kPoolThreads - 1) / kPoolThreads;
  const TIn* h = static_cast<const TIn*>(hidden);
  if (r <= 1)
    embed_pool_kernel<TIn, 1><<<batch, kPoolThreads, 0, st>>>(h, tokens, dim, mask, out, out_bf16);
  else if (r <= 2)
    embed_pool_kernel<TIn, 2><<<batch, kPoolThreads, 0, st>>>(h, tokens, dim, mask, out, out_bf16);
  else if (r <= 4)
    embed_pool_kernel<TIn, 4><<<batch, kPoolThreads, 0, st>>>(h, tokens, dim, mask, out, out_bf16);
  else if (r <= 8)
    embed_pool_kernel<TIn, 8><<<batch, kPoolThreads, 0, st>>>(h, tokens, dim, mask, out, out_bf16);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_embed_pool(int hidden_dtype, const void* hidden, int batch, int tokens, int dim,
                              const uint8_t* mask, int out_dtype, void* out, cudaStream_t st) {
  if (batch <= 0) return cudaSuccess;
  const int out_bf16 = out_dtype == kBF16 ? 1 : 0;
  return hidden_dtype == kBF16
             ? launch_typed<uint16_t>(hidden, batch, tokens, dim, mask, out, out_bf16, st)
             : launch_typed<float>(hidden, batch, tokens, dim, mask, out, out_bf16, st);
}

}  // namespace oprag
