// Device primitives shared by the search kernels: ranking keys, warp-wide
// bitonic sort, per-lane running top-K lists and the list merge.
//
// Ranking follows the TopK definition of Sec. 4.4 (and Op_retrieve, Sec. 3.2):
// higher score first, equal scores broken by the lower chunk id.  A
// (score, id) pair is packed into one 64-bit key whose unsigned order is
// exactly that ranking, so every comparison below is a single integer compare.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

namespace oprag {

constexpr uint64_t kEmptyKey = 0;   // loses to every real candidate

// float -> uint32 whose unsigned order is the float order (-0 folded to +0).
__device__ __forceinline__ uint32_t score_order(float s) {
  uint32_t b = __float_as_uint(s);
  if (b == 0x80000000u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__device__ __forceinline__ float order_score(uint32_t o) {
  uint32_t b = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(b);
}

// key = [score order : 32][~id : 32]; larger key = better rank.
__device__ __forceinline__ uint64_t make_key(float s, uint32_t id) {
  return (static_cast<uint64_t>(score_order(s)) << 32) | static_cast<uint32_t>(~id);
}

__device__ __forceinline__ float key_score(uint64_t k) {
  return order_score(static_cast<uint32_t>(k >> 32));
}

__device__ __forceinline__ uint32_t key_id(uint64_t k) {
  return ~static_cast<uint32_t>(k);
}

// Score a candidate must reach (>=) to possibly enter a list whose worst
// entry is k; -inf while the list is not full.
__device__ __forceinline__ float key_floor(uint64_t k) {
  return k == kEmptyKey ? -INFINITY : key_score(k);
}

__device__ __forceinline__ uint64_t umax64(uint64_t a, uint64_t b) { return a > b ? a : b; }

// Largest 64-bit key of the warp as two 32-bit warp reductions: the largest
// high word, then the largest low word among the lanes that hold it.
__device__ __forceinline__ uint64_t warp_max_key(uint64_t x) {
  const uint32_t hi = __reduce_max_sync(0xffffffffu, static_cast<uint32_t>(x >> 32));
  const uint32_t lo = __reduce_max_sync(
      0xffffffffu, static_cast<uint32_t>(x >> 32) == hi ? static_cast<uint32_t>(x) : 0u);
  return (static_cast<uint64_t>(hi) << 32) | lo;
}
__device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }

// ---------------------------------------------------------------------------
// Warp bitonic sort, descending, of 32*E keys.  Element i lives in lane i/E,
// register i%E.  Strides below E are register swaps, the others lane shuffles.
template <int E>
__device__ __forceinline__ void warp_sort_desc(uint64_t (&v)[E]) {
  const int lane = threadIdx.x & 31;
  constexpr int N = 32 * E;
#pragma unroll
  for (int size = 2; size <= N; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      if (stride < E) {
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int p = e ^ stride;
          if (p > e) {
            const bool desc = (((lane * E + e) & size) == 0);
            const uint64_t a = v[e], b = v[p];
            const bool swap = desc ? (a < b) : (a > b);
            v[e] = swap ? b : a;
            v[p] = swap ? a : b;
          }
        }
      } else {
        const int lmask = stride / E;
        const bool lower = (lane & lmask) == 0;
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const bool desc = (((lane * E + e) & size) == 0);
          const uint64_t o = __shfl_xor_sync(0xffffffffu, v[e], lmask);
          v[e] = (lower == desc) ? umax64(v[e], o) : umin64(v[e], o);
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// a[idx] (0 <= idx < N, N a power of two) for a register array, as a tree of
// selects on the bits of idx, so that the array stays in registers.
template <int N>
__device__ __forceinline__ float reg_select(const float (&a)[N], int idx) {
  static_assert((N & (N - 1)) == 0, "power of two");
  float t[N];
#pragma unroll
  for (int i = 0; i < N; ++i) t[i] = a[i];
#pragma unroll
  for (int w = N / 2; w >= 1; w /= 2) {
    const bool hi = (idx & w) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) t[i] = hi ? t[i + w] : t[i];
  }
  return t[0];
}

// Running top-K of one lane, K <= 32, kept sorted (best first) in registers as
// (score, id) pairs.  Candidates must reach a list in increasing id order (the
// corpus is scanned in id order), so a candidate whose score equals a kept one
// ranks below it and a strict score compare implements the whole ranking.
// Empty slots hold (-inf, ~0u); callers test `s > floor` before push().
constexpr uint32_t kNoId = 0xFFFFFFFFu;

template <int K>
struct RegTopK {
  static constexpr int kStride = K;     // keys per stored list
  float s[K];
  uint32_t id[K];
  float floor;

  __device__ __forceinline__ void init() {
#pragma unroll
    for (int i = 0; i < K; ++i) {
      s[i] = -INFINITY;
      id[i] = kNoId;
    }
    floor = -INFINITY;
  }

  __device__ __forceinline__ bool full() const { return id[K - 1] != kNoId; }

  // k-th best score held (1 <= k <= K); -inf while fewer than k are held.
  __device__ __forceinline__ float kth(int k) const { return reg_select(s, k - 1); }

  __device__ __forceinline__ void push(float v, uint32_t vid) {
    if (v > s[K - 1]) insert(v, vid);
  }

  // Branch-free insertion; a value not above s[K-1] (e.g. -inf) changes nothing.
  __device__ __forceinline__ void insert(float v, uint32_t vid) {
#pragma unroll
    for (int i = K - 1; i > 0; --i) {
      const bool above_prev = v > s[i - 1];
      const bool above_here = v > s[i];
      s[i] = above_prev ? s[i - 1] : (above_here ? v : s[i]);
      id[i] = above_prev ? id[i - 1] : (above_here ? vid : id[i]);
    }
    const bool top = v > s[0];
    s[0] = top ? v : s[0];
    id[0] = top ? vid : id[0];
    floor = s[K - 1];
  }

  __device__ __forceinline__ uint64_t key(int i) const {
    return id[i] == kNoId ? kEmptyKey : make_key(s[i], id[i]);
  }

  __device__ __forceinline__ void store(uint64_t* dst) const {
#pragma unroll
    for (int i = 0; i < K; i += 2)
      *reinterpret_cast<ulonglong2*>(dst + i) = make_ulonglong2(key(i), key(i + 1));
  }

  __device__ __forceinline__ void load(const uint64_t* src) {
#pragma unroll
    for (int i = 0; i < K; i += 2) {
      const ulonglong2 v = *reinterpret_cast<const ulonglong2*>(src + i);
      s[i] = key_floor(v.x);
      id[i] = v.x == kEmptyKey ? kNoId : key_id(v.x);
      s[i + 1] = key_floor(v.y);
      id[i + 1] = v.y == kEmptyKey ? kNoId : key_id(v.y);
    }
    floor = s[K - 1];
  }
};

// ---------------------------------------------------------------------------
// Running top-K of one lane for K in {64,128,256}: candidates that beat the
// current K-th key are appended to a lane-private buffer of 2K keys in global
// memory; the warp compacts a lane's buffer (sort, keep K) once it could
// overflow within the next 32 pushes.  Callers push at most 32 times between
// calls to sync().
template <int K>
struct BufTopK {
  static constexpr int kCap = 2 * K;
  static constexpr int kStride = kCap;
  static constexpr int kE = kCap / 32;
  uint64_t* buf;
  int count;
  uint64_t worst;      // K-th best key once K keys were kept, else empty
  float floor;

  __device__ __forceinline__ void init(uint64_t* b) {
    buf = b;
    count = 0;
    worst = kEmptyKey;
    floor = -INFINITY;
  }

  __device__ __forceinline__ void push(float s, uint32_t id) {
    const uint64_t key = make_key(s, id);
    if (key > worst) buf[count++] = key;
  }

  // Warp-collective; lanes with active == false own no buffer.  final == true
  // sorts every active lane's buffer and leaves its best K keys (padded with
  // empty keys) in buf[0..K).
  __device__ void sync(bool final, bool active) {
    const int lane = threadIdx.x & 31;
    __syncwarp();
    uint32_t need = __ballot_sync(0xffffffffu, active && (final || count > kCap - 32));
    while (need) {
      const int src = __ffs(need) - 1;
      need &= need - 1;
      uint64_t* b = reinterpret_cast<uint64_t*>(
          __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(buf), src));
      const int c = __shfl_sync(0xffffffffu, count, src);
      uint64_t v[kE];
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        const int i = lane * kE + e;
        v[e] = i < c ? b[i] : kEmptyKey;
      }
      warp_sort_desc<kE>(v);
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        const int i = lane * kE + e;
        if (i < K) b[i] = v[e];
      }
      const uint64_t kth = __shfl_sync(0xffffffffu, v[(K - 1) % kE], (K - 1) / kE);
      if (lane == src) {
        count = c < K ? c : K;
        // Every kept key beats the old floor, so the floor only rises.
        if (c >= K) worst = kth;
        floor = key_floor(worst);
      }
      __syncwarp();
    }
  }
};

// ---------------------------------------------------------------------------
// Warp-cooperative merge of sorted key lists into the best KP keys, using a
// shared-memory buffer of 2*KP keys.  Lists are read only while their keys can
// still enter (they are sorted, so the first key that cannot enter ends them).
template <int KP>
struct WarpMerger {
  static constexpr int kCap = 2 * KP;
  static constexpr int kE = kCap / 32;
  uint64_t* sbuf;      // kCap keys in shared memory
  int count;           // warp-uniform
  uint64_t worst;      // warp-uniform: k-th best once known
  int k;

  __device__ __forceinline__ void init(uint64_t* s, int k_) {
    sbuf = s;
    count = 0;
    worst = kEmptyKey;
    k = k_;
  }

  // Not inlined: the merges offer keys from unrolled loops, and one copy of
  // the sort per offer made their code outgrow the instruction cache.
  __device__ __noinline__ void compact() {
    const int lane = threadIdx.x & 31;
    __syncwarp();
    uint64_t v[kE];
#pragma unroll
    for (int e = 0; e < kE; ++e) {
      const int i = lane * kE + e;
      v[e] = i < count ? sbuf[i] : kEmptyKey;
    }
    warp_sort_desc<kE>(v);
    __syncwarp();
#pragma unroll
    for (int e = 0; e < kE; ++e) {
      const int i = lane * kE + e;
      if (i < KP) sbuf[i] = v[e];
    }
    uint64_t mine = kEmptyKey;
#pragma unroll
    for (int e = 0; e < kE; ++e)
      if (e == (k - 1) % kE) mine = v[e];
    const uint64_t kth = __shfl_sync(0xffffffffu, mine, (k - 1) / kE);
    if (count >= k) worst = kth;
    count = count < KP ? count : KP;
    __syncwarp();
  }

  // Offers one sorted list of len keys (stride 1).
  __device__ void offer_list(const uint64_t* list, int len) {
    const int lane = threadIdx.x & 31;
    for (int off = 0; off < len; off += 32) {
      const uint64_t key = (off + lane < len) ? list[off + lane] : kEmptyKey;
      const bool pass = key > worst;
      const uint32_t m = __ballot_sync(0xffffffffu, pass);
      if (m == 0) break;
      if (count > kCap - 32) compact();
      if (pass) sbuf[count + __popc(m & ((1u << lane) - 1u))] = key;
      count += __popc(m);
    }
  }

  // Sorts what is kept; afterwards sbuf[0..k) holds the answer (empty keys pad).
  __device__ void finish() { compact(); }
};

// ---------------------------------------------------------------------------
// Bounded waits.  Every spin on an mbarrier gives up after ~2^31 cycles (about
// a second), records the failure in a device-wide error word and returns false,
// so that a lost arrival ends the kernel instead of hanging the GPU.
constexpr int64_t kWaitLimitCycles = 1ll << 31;

enum DeviceError : int {
  kDevErrNone = 0,
  kDevErrWaitTimeout = 1,
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Longest time (ns) a waiting thread stays suspended in one try_wait before it
// looks at the abort word and the clock again; the thread resumes as soon as
// the phase completes.  Without the hint the system's short default made the
// waiting warps (an epilogue set waits about half of the time) poll, taking
// issue slots from the producer and MMA warps: measured on GB300, 1M x 768 with
// 2048 queries and k = 100, main pass 1905 instead of 2061 us; 32768 x 1024
// with 4096 queries and k = 10, 199 instead of 211 us; one query, no slower.
constexpr int kSuspendHintNs = 20000;

// kCluster: acquire at cluster scope (the phase was completed by arrivals
// from the other CTA of a cluster).
template <bool kCluster = false>
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  if constexpr (kCluster) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity), "n"(kSuspendHintNs)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity), "n"(kSuspendHintNs)
        : "memory");
  }
  return ok != 0;
}

// Non-blocking probe of a phase (mbarrier.test_wait returns at once, where
// try_wait may suspend the thread until the phase completes).
template <bool kCluster = false>
__device__ __forceinline__ bool mbar_probe(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  if constexpr (kCluster) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
  }
  return ok != 0;
}

// Waits for the phase with the given parity to complete.  Gives up when the
// CTA-wide abort word is set or `limit` cycles pass (then sets both).  A limit
// below the default (a test shortening it) spins on non-blocking probes, so
// that even a wait that hardware would complete within its suspend time runs
// out.
template <bool kCluster = false>
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          int* dev_err, long long limit = kWaitLimitCycles) {
  if (limit < kWaitLimitCycles) {
    const long long t0 = clock64();
    while (!mbar_probe<kCluster>(bar, parity)) {
      if (*abort_flag) return false;
      if (clock64() - t0 > limit) {
        *abort_flag = 1;
        atomicExch(dev_err, static_cast<int>(kDevErrWaitTimeout));
        return false;
      }
    }
    return true;
  }
  if (mbar_test<kCluster>(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_test<kCluster>(bar, parity)) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) {
      *abort_flag = 1;
      atomicExch(dev_err, static_cast<int>(kDevErrWaitTimeout));
      return false;
    }
  }
}

}  // namespace oprag
