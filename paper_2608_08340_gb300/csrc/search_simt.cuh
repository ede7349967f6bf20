// SIMT streaming search: dense inner-product scoring (Sec. 4.4, "vectorized
// matrix operations over the embedding matrix") with the running partial top-k
// fused in (Sec. 4.4 / Sec. 7: partial selection instead of a full sort).
//
// Used for fp32 indices (whose scores must be exact fp32 FMA sums, which the
// bf16 tensor path cannot give) and for bf16 searches with very few queries,
// where the pass is a pure HBM stream and tensor cores buy nothing.
//
// Layout: each warp owns a contiguous range of corpus rows and walks it one
// row at a time with 16-byte loads spread over its 32 lanes (4 rows in flight
// per warp for memory-level parallelism).  A chunk of QC <= 8 queries sits in
// shared memory as fp32.  After a butterfly reduction every lane holds the QC
// scores of the row; lane j keeps the running top-K of query j.  The eight
// warps' lists are merged in shared memory into one list per (CTA, query);
// the merge kernel reduces those across CTAs.
#pragma once
#include "common.cuh"
#include "internal.h"

namespace oprag {
namespace simt {

constexpr int kSimtWarps = 8;
constexpr int kRowsInFlight = 4;

template <typename T>
struct Vec;

template <>
struct Vec<float> {
  static constexpr int kElems = 4;
  __device__ __forceinline__ static void unpack(const uint4& v, float (&x)[4]) {
    x[0] = __uint_as_float(v.x);
    x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z);
    x[3] = __uint_as_float(v.w);
  }
};

template <>
struct Vec<__nv_bfloat16> {
  static constexpr int kElems = 8;
  __device__ __forceinline__ static void unpack(const uint4& v, float (&x)[8]) {
    x[0] = __uint_as_float(v.x << 16);
    x[1] = __uint_as_float(v.x & 0xFFFF0000u);
    x[2] = __uint_as_float(v.y << 16);
    x[3] = __uint_as_float(v.y & 0xFFFF0000u);
    x[4] = __uint_as_float(v.z << 16);
    x[5] = __uint_as_float(v.z & 0xFFFF0000u);
    x[6] = __uint_as_float(v.w << 16);
    x[7] = __uint_as_float(v.w & 0xFFFF0000u);
  }
};

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}

// Lane-private top-K with a uniform interface over the register and the
// buffered variants.
template <int K, bool kBuf = (K > 32)>
struct LaneList;

template <int K>
struct LaneList<K, false> {
  RegTopK<K> t;
  __device__ __forceinline__ void init(uint64_t*) { t.init(); }
  __device__ __forceinline__ float floor() const { return t.floor; }
  __device__ __forceinline__ void push(float s, uint32_t id) { t.push(s, id); }
  __device__ __forceinline__ void sync(bool, bool) {}
  // Writes the sorted best K keys to dst.
  __device__ __forceinline__ void emit(uint64_t* dst, bool active) {
    if (active) t.store(dst);
  }
};

template <int K>
struct LaneList<K, true> {
  BufTopK<K> t;
  __device__ __forceinline__ void init(uint64_t* b) { t.init(b); }
  __device__ __forceinline__ float floor() const { return t.floor; }
  __device__ __forceinline__ void push(float s, uint32_t id) { t.push(s, id); }
  __device__ __forceinline__ void sync(bool final, bool active) { t.sync(final, active); }
  __device__ __forceinline__ void emit(uint64_t* dst, bool active) {
    t.sync(true, active);
    if (active)
      for (int i = 0; i < K; ++i) dst[i] = t.buf[i];
  }
};

// grid = (CTAs over corpus rows, ceil(q / QC) query chunks), 256 threads.
// scratch layout: [chunk][cta][QC][K] CTA lists, then (buffered K only)
// [chunk][cta][warp][QC][2K] lane buffers.
template <typename T, int QC, int K>
__global__ void __launch_bounds__(kSimtWarps * 32)
simt_search_kernel(const T* __restrict__ E, int64_t n, int d, const T* __restrict__ Q, int q,
                   int k, Fusion fu, uint64_t* __restrict__ cta_lists,
                   uint64_t* __restrict__ lane_bufs) {
  constexpr int VE = Vec<T>::kElems;
  constexpr int kMergeCap = 2 * (K < 32 ? 32 : K);
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* qs = reinterpret_cast<float*>(smem_raw);                          // QC x d
  uint64_t* wl = reinterpret_cast<uint64_t*>(smem_raw + sizeof(float) * QC * d);  // 8 x QC x K
  uint64_t* mbuf = wl + kSimtWarps * QC * K;                                 // QC x kMergeCap

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int chunk = blockIdx.y;
  const int q0 = chunk * QC;
  const int nq = min(QC, q - q0);

  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  for (int i = threadIdx.x; i < QC * d; i += blockDim.x) {
    const int qq = i / d, j = i % d;
    qs[i] = qq < nq ? to_f32<T>(Q[static_cast<int64_t>(q0 + qq) * d + j]) : 0.f;
  }
  __syncthreads();

  // Rows of this warp: a contiguous slice of the corpus.
  const int64_t total_warps = static_cast<int64_t>(gridDim.x) * kSimtWarps;
  const int64_t gw = static_cast<int64_t>(blockIdx.x) * kSimtWarps + warp;
  const int64_t r_begin = gw * n / total_warps;
  const int64_t r_end = (gw + 1) * n / total_warps;

  const bool active = lane < nq;
  const int qg = q0 + (active ? lane : 0);
  float inv_max = 0.f;
  const float* brow = nullptr;
  if (fu.bm25 != nullptr && active) {
    const float m = fu.bm25_max[qg];
    inv_max = m > 0.f ? 1.f / m : 0.f;
    brow = fu.bm25 + static_cast<int64_t>(qg) * fu.ld;
  }

  LaneList<K> list;
  {
    uint64_t* my_buf = nullptr;
    if (K > 32 && active)
      my_buf = lane_bufs +
               (((static_cast<int64_t>(chunk) * gridDim.x + blockIdx.x) * kSimtWarps + warp) * QC +
                lane) * (2 * K);
    list.init(my_buf);
  }

  const int nvec = d / VE;                     // 16-byte vectors per row
  int since_sync = 0;
  for (int64_t r0 = r_begin; r0 < r_end; r0 += kRowsInFlight) {
    float acc[kRowsInFlight][QC];
#pragma unroll
    for (int rr = 0; rr < kRowsInFlight; ++rr)
#pragma unroll
      for (int qq = 0; qq < QC; ++qq) acc[rr][qq] = 0.f;

    for (int v = lane; v < nvec; v += 32) {
      uint4 raw[kRowsInFlight];
#pragma unroll
      for (int rr = 0; rr < kRowsInFlight; ++rr) {
        const int64_t r = r0 + rr;
        raw[rr] = r < r_end ? __ldcs(reinterpret_cast<const uint4*>(E + r * d) + v)
                            : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int rr = 0; rr < kRowsInFlight; ++rr) {
        float x[VE];
        Vec<T>::unpack(raw[rr], x);
#pragma unroll
        for (int qq = 0; qq < QC; ++qq) {
          const float* qv = qs + qq * d + v * VE;
#pragma unroll
          for (int e = 0; e < VE; e += 4) {
            const float4 w = *reinterpret_cast<const float4*>(qv + e);
            acc[rr][qq] = fmaf(x[e], w.x, acc[rr][qq]);
            acc[rr][qq] = fmaf(x[e + 1], w.y, acc[rr][qq]);
            acc[rr][qq] = fmaf(x[e + 2], w.z, acc[rr][qq]);
            acc[rr][qq] = fmaf(x[e + 3], w.w, acc[rr][qq]);
          }
        }
      }
    }
    // Butterfly: every lane ends with the full sums.
#pragma unroll
    for (int rr = 0; rr < kRowsInFlight; ++rr)
#pragma unroll
      for (int qq = 0; qq < QC; ++qq)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
          acc[rr][qq] += __shfl_xor_sync(0xffffffffu, acc[rr][qq], o);

#pragma unroll
    for (int rr = 0; rr < kRowsInFlight; ++rr) {
      const int64_t r = r0 + rr;
      float s = 0.f;
#pragma unroll
      for (int qq = 0; qq < QC; ++qq)
        if (qq == lane) s = acc[rr][qq];
      if (active && r < r_end) {
        if (brow != nullptr) s = fmaf(fu.alpha, s, (1.f - fu.alpha) * (brow[r] * inv_max));
        if (s >= list.floor()) list.push(s, static_cast<uint32_t>(r));
      }
    }
    since_sync += kRowsInFlight;
    if (since_sync >= 32 - kRowsInFlight) {
      list.sync(false, active);
      since_sync = 0;
    }
  }

  // Lists of the eight warps -> shared memory -> one list per (CTA, query).
  list.emit(wl + (warp * QC + (active ? lane : 0)) * K, active);
  __syncthreads();
  if (warp < nq) {
    WarpMerger<(K < 32 ? 32 : K)> m;
    m.init(mbuf + warp * kMergeCap, k);
    for (int w = 0; w < kSimtWarps; ++w) m.offer_list(wl + (w * QC + warp) * K, k);
    m.finish();
    uint64_t* dst = cta_lists +
                    ((static_cast<int64_t>(chunk) * gridDim.x + blockIdx.x) * QC + warp) * K;
    for (int i = lane; i < K; i += 32) dst[i] = i < k ? m.sbuf[i] : kEmptyKey;
  }
}

template <typename T, int QC, int K>
size_t simt_smem(int d) {
  return sizeof(float) * QC * d + sizeof(uint64_t) * kSimtWarps * QC * K +
         sizeof(uint64_t) * QC * 2 * (K < 32 ? 32 : K);
}


template <typename T, int QC, int K>
cudaError_t launch_t(const void* E, const void* Q, const SearchShape& s, const Fusion& fu,
                     void* scratch, int grid, ListSet* lists, cudaStream_t st) {
  const int chunks = (s.q + QC - 1) / QC;
  uint64_t* cta_lists = static_cast<uint64_t*>(scratch);
  uint64_t* lane_bufs = cta_lists + static_cast<size_t>(chunks) * grid * QC * K;
  const size_t smem = simt_smem<T, QC, K>(s.d);
  cudaError_t e = cudaFuncSetAttribute(simt_search_kernel<T, QC, K>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  simt_search_kernel<T, QC, K><<<dim3(grid, chunks), kSimtWarps * 32, smem, st>>>(
      static_cast<const T*>(E), s.n, s.d, static_cast<const T*>(Q), s.q, s.k, fu, cta_lists,
      lane_bufs);
  lists->keys = cta_lists;
  lists->P = grid;
  lists->TH = QC;
  lists->stride = K;
  lists->klen = K;
  return cudaGetLastError();
}

template <typename T, int QC>
cudaError_t launch_qc(const void* E, const void* Q, const SearchShape& s, const Fusion& fu,
                      void* scratch, int grid, ListSet* lists, cudaStream_t st) {
  switch (list_len_for(s.k)) {
    case 8: return launch_t<T, QC, 8>(E, Q, s, fu, scratch, grid, lists, st);
    case 16: return launch_t<T, QC, 16>(E, Q, s, fu, scratch, grid, lists, st);
    case 32: return launch_t<T, QC, 32>(E, Q, s, fu, scratch, grid, lists, st);
    case 128: return launch_t<T, QC, 128>(E, Q, s, fu, scratch, grid, lists, st);
    default: return launch_t<T, QC, 256>(E, Q, s, fu, scratch, grid, lists, st);
  }
}

cudaError_t launch_f32(int qc, const void* E, const void* Q, const SearchShape& s, const Fusion& fu,
                       void* scratch, int grid, ListSet* lists, cudaStream_t st);
cudaError_t launch_bf16(int qc, const void* E, const void* Q, const SearchShape& s,
                        const Fusion& fu, void* scratch, int grid, ListSet* lists,
                        cudaStream_t st);

}  // namespace simt
}  // namespace oprag
