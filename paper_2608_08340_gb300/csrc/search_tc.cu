// Host planning for the tensor-core search kernel of search_tc.cuh: tile
// size, persistent grid, slot bookkeeping, scratch size and TMA descriptors.
#include "search_tc.cuh"

namespace oprag {

using namespace tc;

namespace {

// ----------------------------------------------------------------- host

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &qres) == cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// Row-major rows x d bf16 matrix, boxes of 64 columns x box_rows rows, 128-byte swizzle;
// rows past the end read as zero.
bool make_map(CUtensorMap* m, const void* base, int64_t rows, int d, int box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

int gcd_int(int a, int b) {
  while (b) {
    const int t = a % b;
    a = b;
    b = t;
  }
  return a;
}

}  // namespace

TcPlan tc_plan(const SearchShape& s, int num_sms, int force_block_n) {
  TcPlan pl{};
  pl.qt = (s.q + kBlockM - 1) / kBlockM;
  int bn = 256;
  if (force_block_n == 64 || force_block_n == 256) {
    bn = force_block_n;
  } else {
    // Small query batches leave few units: cut the corpus finer so that every
    // SM gets several units.
    const int64_t units256 = static_cast<int64_t>(pl.qt) * ((s.n + 255) / 256);
    if (units256 < 4LL * num_sms) bn = 64;
  }
  pl.block_n = bn;
  const int64_t nt = (s.n + bn - 1) / bn;
  const int64_t units = nt * pl.qt;
  pl.grid = static_cast<int>(units < num_sms ? units : num_sms);
  if (pl.grid < 1) pl.grid = 1;
  const int g = gcd_int(pl.grid, pl.qt);
  pl.slots = pl.qt / g;
  pl.P = pl.grid / g;
  pl.stages = bn == 64 ? stages_for<64>() : stages_for<256>();
  pl.smem = bn == 64 ? smem_for<64>() : smem_for<256>();
  return pl;
}

size_t tc_scratch_bytes(const SearchShape& s, const TcPlan& pl) {
  const int K = list_len_for(s.k);
  const int stride = K > 32 ? 2 * K : K;
  const size_t rows = static_cast<size_t>(pl.qt) * pl.P * kBlockM;
  size_t bytes = rows * stride * sizeof(uint64_t);
  if (K > 32) bytes += rows * (sizeof(uint64_t) + sizeof(int));
  return bytes;
}

cudaError_t launch_tc_search(const void* E, const void* Q, const SearchShape& s, const Fusion& fu,
                             const TcPlan& pl, void* scratch, int* dev_err, ListSet* lists,
                             cudaStream_t st) {
  CUtensorMap mq, me;
  if (!make_map(&mq, Q, s.q, s.d, kBlockM) || !make_map(&me, E, s.n, s.d, pl.block_n))
    return cudaErrorInvalidValue;
  const int K = list_len_for(s.k);
  const int stride = K > 32 ? 2 * K : K;
  const size_t rows = static_cast<size_t>(pl.qt) * pl.P * kBlockM;
  TcParams prm{};
  prm.n = s.n;
  prm.d = s.d;
  prm.q = s.q;
  prm.k = s.k;
  prm.qt = pl.qt;
  prm.units = static_cast<int64_t>(pl.qt) * ((s.n + pl.block_n - 1) / pl.block_n);
  prm.g = gcd_int(pl.grid, pl.qt);
  prm.P = pl.P;
  prm.slots = pl.slots;
  prm.kblocks = (s.d + kBlockK - 1) / kBlockK;
  prm.fu = fu;
  prm.lists = static_cast<uint64_t*>(scratch);
  prm.meta_worst = prm.lists + rows * stride;
  prm.meta_count = reinterpret_cast<int*>(prm.meta_worst + (K > 32 ? rows : 0));
  prm.dev_err = dev_err;
  lists->keys = prm.lists;
  lists->P = pl.P;
  lists->TH = kBlockM;
  lists->stride = stride;
  const bool hybrid = fu.bm25 != nullptr;
  if (pl.block_n == 64) return launch_bn64(mq, me, prm, pl.grid, hybrid, st);
  return hybrid ? launch_bn256_fused(mq, me, prm, pl.grid, st)
                : launch_bn256_dense(mq, me, prm, pl.grid, st);
}

}  // namespace oprag
