// Restoration round r (Sec. 4.3), first half, on the tensor cores: the gain inner products
//   t_ij = (y~_i - z~_j) . g~_i = c_i - z~_j . g~_i,   c_i = y~_i . g~_i      (Eq. 14/15)
// for every candidate row i and candidate block j of a head, without the P_ij factor.
//
// z~_j . g~_i is a [|P| x 64] x [64 x |P|] product per head.  Both operands are fp32; each
// is held as the sum of three bf16 terms (hi + mid + lo, written by the kernels that
// produce g~ and z~), and the product is accumulated in fp32 TMEM from the six term
// products whose size is at least 2^-16 of hi.hi:
//   mid.mid + hi.lo + lo.hi + hi.mid + mid.hi + hi.hi      (smallest first)
// The three dropped products are below 2^-23 of |z~||g~| together, the size of the fp32
// rounding of the dot product itself.
//
// One CTA per 128 x 128 tile of (i, j) of one head, 128 threads:
//   thread 0   TMA of the six 128 x 64 bf16 term tiles (128-byte swizzle) on one mbarrier;
//   warp 0     converged MMA warp, one elected lane issues 6 x 4 tcgen05.mma M128 N128 K16
//              (A = g~ terms, B = z~ terms, both K-major from shared memory) and commits;
//   warps 0-3  epilogue: tcgen05.ld of the accumulator rows (warp w: rows 32w..32w+31),
//              t = c_i - acc into shared memory (the operand tiles are free by then) as
//              four 32-column boxes in the 128-byte-swizzled layout, which thread 0 writes
//              to t with TMA bulk tensor stores (rows past nb and columns past the row
//              stride are clipped by the copy; rows past |P| are never read).
// Every mbarrier wait is bounded; a wait that gives up records RESS_ETIMEOUT, lets copies
// and MMAs already issued finish (again bounded), frees TMEM and returns.

#include <cudaTypedefs.h>

#include "ress_internal.cuh"
#include "sm100_ptx.cuh"

namespace ress {
using namespace ptx;

namespace {

constexpr int kGainThreads = 128;
constexpr int kGainTile = 128;                     // rows i and blocks j per CTA
constexpr uint32_t kTermBytes = kGainTile * 128;   // 128 x 64 bf16
constexpr uint32_t kGainCols = 128;                // TMEM columns: one fp32 128 x 128 tile
constexpr uint64_t kGainWaitNs = 2000000000ull;    // 2 s per wait
constexpr uint64_t kGainDrainNs = 200000000ull;    // 0.2 s to drain after an abort

struct __align__(1024) GainSmem {
  uint8_t A[3][kTermBytes];  // g~ terms (hi, mid, lo) of rows i0 .. i0 + 127
  uint8_t B[3][kTermBytes];  // z~ terms of blocks j0 .. j0 + 127
  uint64_t full, done;
  uint32_t tmem_base;
  int abort;
};

struct GainParams {
  int nb, ncand, ld, round;
  float rho;
  const float* cdot;  // [H, nb]
  float* t;           // [H, nb, ld]
  uint32_t* status;
  Budgets bud;
};

// (A term, B term) of product q of the six, smallest first: 4 bits per q.
constexpr uint32_t kTermA = 0x010201u;  // q = 0..5 -> 1, 0, 2, 0, 1, 0
constexpr uint32_t kTermB = 0x001021u;  // q = 0..5 -> 1, 2, 0, 1, 0, 0

// Bounded wait by a whole warp (all lanes test once; otherwise lane 0 polls and broadcasts).
__device__ __forceinline__ bool gain_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          uint64_t limit_ns) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, limit_ns) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

__global__ void __launch_bounds__(kGainThreads)
    k_gain(const __grid_constant__ CUtensorMap tmG, const __grid_constant__ CUtensorMap tmZ,
           const __grid_constant__ CUtensorMap tmT, const GainParams p) {
  const int h = blockIdx.z, i0 = blockIdx.y * kGainTile, j0 = blockIdx.x * kGainTile;
  if (swap_count(p.bud.c[h], p.ncand, p.round, p.rho) <= 0) return;
  extern __shared__ uint8_t smem_raw[];
  GainSmem& S = *reinterpret_cast<GainSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;

  if (threadIdx.x == 0) {
    mbar_init(&S.full, 1);
    mbar_init(&S.done, 1);
    S.abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&tmG);
    prefetch_tensormap(&tmZ);
    prefetch_tensormap(&tmT);
  }
  if (warp == 0) tmem_alloc(&S.tmem_base, kGainCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = S.tmem_base;

  bool issued = false;  // warp 0: MMAs went out (their completion must be awaited)
  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(&S.full, 6 * kTermBytes);
#pragma unroll
      for (int s = 0; s < 3; ++s) {
        tma_load_4d(S.A[s], &tmG, &S.full, 0, i0, h, s);
        tma_load_4d(S.B[s], &tmZ, &S.full, 0, j0, h, s);
      }
    }
    __syncwarp();
    const bool leader = elect_one();
    if (__popc(__ballot_sync(0xffffffffu, leader)) != 1) {  // exactly one issuing lane
      if (lane == 0) {
        flag_status(p.status, kStatusBadRow);
        *abort = 1;
      }
    } else if (gain_wait(&S.full, 0, abort, kGainWaitNs)) {
      tc_fence_after();
      const uint32_t idesc = idesc_bf16_f32(kGainTile, kGainTile, false);
      if (leader) {
#pragma unroll
        for (int q = 0; q < 6; ++q) {
          const uint32_t a = smem_u32(S.A[(kTermA >> (4 * q)) & 0xF]);
          const uint32_t b = smem_u32(S.B[(kTermB >> (4 * q)) & 0xF]);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_bf16_ss(tmem, sdesc_sw128(a + 32 * k), sdesc_sw128(b + 32 * k), idesc,
                        (q > 0 || k > 0) ? 1u : 0u);
        }
        mma_commit(&S.done);
      }
      __syncwarp();
      issued = true;
    } else if (lane == 0) {
      flag_status(p.status, kStatusTimeout);
      *abort = 1;
    }
    if (!issued) {  // the copies must land before the shared memory goes away
      volatile int no_abort = 0;
      if (lane == 0) mbar_wait(&S.full, 0, &no_abort, kGainDrainNs);
      __syncwarp();
    }
  }

  // ---- epilogue: warp w holds rows 32w .. 32w + 31 of the tile (TMEM lanes) ----------
  bool ok = gain_wait(&S.done, 0, abort, kGainWaitNs);
  if (!ok && lane == 0 && !*abort) {
    flag_status(p.status, kStatusTimeout);
    *abort = 1;
  }
  if (ok) {
    tc_fence_after();
    const int r = 32 * warp + lane;  // row of the tile = TMEM lane
    const int i = i0 + r;
    const float c = i < p.nb ? p.cdot[(int64_t)h * p.nb + i] : 0.f;
    uint8_t* stage = &S.A[0][0];  // 4 boxes of 128 rows x 32 fp32, 16 KB each
#pragma unroll 1
    for (int q = 0; q < kGainTile / 32; ++q) {
      uint32_t v[32];
      RESS_TMEM_LD32(tmem + ((uint32_t)(32 * warp) << 16) + 32 * q, v);
      uint8_t* row = stage + q * 16384 + r * 128;
#pragma unroll
      for (int k = 0; k < 8; ++k)  // 16-byte chunk k of the row goes to chunk k ^ (r mod 8)
        *reinterpret_cast<float4*>(row + ((k ^ (r & 7)) << 4)) =
            make_float4(c - __uint_as_float(v[4 * k]), c - __uint_as_float(v[4 * k + 1]),
                        c - __uint_as_float(v[4 * k + 2]), c - __uint_as_float(v[4 * k + 3]));
    }
    fence_proxy_async_smem();
  }
  __syncthreads();
  if (ok && threadIdx.x == 0) {
#pragma unroll 1
    for (int q = 0; q < kGainTile / 32; ++q)
      if (j0 + 32 * q < p.ld) tma_store_3d(&tmT, &S.A[0][0] + q * 16384, j0 + 32 * q, i0, h);
    bulk_commit();
    bulk_wait_read_all();  // the boxes are read before the shared memory goes away
  }
  if (warp == 0 && issued && !ok) {  // MMAs still running: let them finish before the free
    volatile int no_abort = 0;
    if (lane == 0) mbar_wait(&S.done, 0, &no_abort, kGainDrainNs);
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kGainCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 gain_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* q = nullptr;
    cudaDriverEntryPointQueryResult r;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &q, 12000, cudaEnableDefault,
                                         &r) == cudaSuccess &&
        r == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(q);
  }
  return fn;
}

// bf16 [3][H][nb][64] viewed as {64, nb, H, 3}; box {64, 128, 1, 1}, 128-byte swizzle.
// Rows past nb read as zeros.
bool make_term_map(CUtensorMap* m, const void* base, int nb, int H) {
  auto fn = gain_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {64, (cuuint64_t)nb, (cuuint64_t)H, 3};
  cuuint64_t strides[3] = {128, (cuuint64_t)nb * 128, (cuuint64_t)H * nb * 128};
  cuuint32_t box[4] = {64, (cuuint32_t)kGainTile, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// t: fp32 [H][nb][ld] viewed as {ld, nb, H}; box {32, 128, 1}, 128-byte swizzle.
bool make_gain_out_map(CUtensorMap* m, void* base, int nb, int H, int ld) {
  auto fn = gain_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)ld, (cuuint64_t)nb, (cuuint64_t)H};
  cuuint64_t strides[2] = {(cuuint64_t)ld * 4, (cuuint64_t)nb * ld * 4};
  cuuint32_t box[3] = {32, (cuuint32_t)kGainTile, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_gain(const SelectArgs& a, int round, float rho, cudaStream_t st) {
  const Shape& s = a.s;
  if (s.ncand <= 0) return cudaSuccess;
  CUtensorMap tg, tz, tt;
  if (!make_term_map(&tg, a.ws + a.L.gsplit, s.nb, s.H) ||
      !make_term_map(&tz, a.ws + a.L.zsplit, s.nb, s.H) ||
      !make_gain_out_map(&tt, a.ws + a.L.t, s.nb, s.H, s.ld))
    return cudaErrorInvalidValue;
  GainParams p;
  p.nb = s.nb;
  p.ncand = s.ncand;
  p.ld = s.ld;
  p.round = round;
  p.rho = rho;
  p.cdot = (const float*)(a.ws + a.L.cdot);
  p.t = (float*)(a.ws + a.L.t);
  p.status = (uint32_t*)(a.ws + a.L.status);
  for (int h = 0; h < RESS_MAX_HEADS; ++h) p.bud.c[h] = a.c[h];
  const size_t smem = sizeof(GainSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(k_gain, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int tiles = (s.ncand + kGainTile - 1) / kGainTile;
  k_gain<<<dim3(tiles, tiles, s.H), kGainThreads, smem, st>>>(tg, tz, tt, p);
  return cudaGetLastError();
}

}  // namespace ress
