// What the attention sublayer adds to the residual stream (Sec. 3), on the tensor cores:
//   residual update:   y = x + O W_o^T                 (bf16 in and out, fp32 accumulation)
//   token-level drift: drift[b] = sum_{t in block b} ||W_o (O_a[t] - O_b[t])||^2
// O is [N, K] with K = H * 64 (the concatenated head outputs), W_o is [d_model, K] (Linear
// weight, out x in), x and y are [N, d_model].
//
// One tile = 128 tokens x 256 output channels, reduced over K in 64-wide slices through a
// three-stage TMA ring (128-byte swizzle, both operands K-major).  192 threads:
//   warp 0     TMA of the O and W_o slices (the drift variant loads O_a and O_b slices);
//   warp 1     TMEM owner; one elected lane of the converged warp issues per slice 4 x
//              tcgen05.mma M128 N256 K16 (the drift variant: 4 into each of two accumulators);
//   warps 2-5  epilogue, row r = TMEM lane: residual update: the tile's x (loaded by TMA into
//              a swizzled staging area) plus the accumulator, rounded to bf16 in place and
//              written out by TMA bulk stores; drift: the squared difference of the two
//              accumulators summed over the row's channels, then over each block's 64 rows
//              in a fixed order.
// The residual update runs persistent CTAs over the tiles with two TMEM accumulators, so a
// tile's epilogue overlaps the next tile's MMAs; the drift variant gives each CTA one
// 128-token stripe and walks its channel tiles in order.
// Every mbarrier wait is bounded; a wait that gives up records RESS_ETIMEOUT, makes the CTA
// leave its loops together, lets copies and MMAs already issued finish (again bounded), frees
// TMEM and returns.

#include <cudaTypedefs.h>

#include "ress_internal.cuh"
#include "sm100_ptx.cuh"

namespace ress {
using namespace ptx;

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

namespace {

constexpr int kOThreads = 192;
constexpr int kOM = 128;                      // tokens per tile
constexpr int kON = 256;                      // output channels per tile
constexpr int kOStages = 3;
constexpr uint32_t kABytes = kOM * 128;       // 128 x 64 bf16
constexpr uint32_t kBBytes = kON * 128;       // 256 x 64 bf16
constexpr uint32_t kOCols = 512;              // TMEM: two 128 x 256 fp32 accumulators
constexpr uint64_t kOWaitNs = 2000000000ull;  // 2 s per wait
constexpr uint64_t kODrainNs = 200000000ull;  // 0.2 s to drain after an abort

enum { kResidual = 0, kDrift = 1 };

// Shared-memory layout.  Residual: A[3] | B[3] | X (4 boxes of 128 x 64 bf16).
// Drift: A[3] | A2[3] | B[3].
constexpr uint32_t kOffA = 0;
constexpr uint32_t kOffB = kOStages * kABytes;                 // residual
constexpr uint32_t kOffX = kOffB + kOStages * kBBytes;
constexpr uint32_t kOffA2 = kOStages * kABytes;                // drift
constexpr uint32_t kOffB2 = kOffA2 + kOStages * kABytes;
constexpr uint32_t kOData = kOffX + 4 * 16384;                 // the larger of the two layouts
static_assert(kOffB2 + kOStages * kBBytes <= kOData, "drift layout fits the residual one");

struct OCtl {
  float rowsum[kOM];
  uint64_t full[kOStages], empty[kOStages], acc_full[2], acc_empty[2], x_full;
  uint32_t tmem_base;
  int abort;
};

struct OParams {
  int N, K, Dm, nb;
  int mtiles, ntiles;
  bool has_x;
  float* drift;
  uint32_t* status;
};

__device__ __forceinline__ bool o_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, kOWaitNs) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

__device__ __forceinline__ void o_give_up(OCtl& C, uint32_t* status) {
  flag_status(status, kStatusTimeout);
  *reinterpret_cast<volatile int*>(&C.abort) = 1;
}

// Named barrier of the four epilogue warps that also ANDs a flag across them.
__device__ __forceinline__ bool o_epi_sync_and(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, 128, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void o_epi_sync() { asm volatile("bar.sync 2, 128;" ::: "memory"); }

template <int MODE>
__device__ __forceinline__ int tiles_of_cta(const OParams& p) {
  if (MODE == kDrift) return p.ntiles;
  const int total = p.mtiles * p.ntiles;
  return blockIdx.x < total ? (total - 1 - blockIdx.x) / gridDim.x + 1 : 0;
}
template <int MODE>
__device__ __forceinline__ void tile_coords(const OParams& p, int k, int& mt, int& nt) {
  if (MODE == kDrift) {
    mt = blockIdx.x;
    nt = k;
  } else {  // consecutive tiles share their token stripe, so O slices are re-read from L2
    const int t = blockIdx.x + k * gridDim.x;
    mt = t / p.ntiles;
    nt = t % p.ntiles;
  }
}

template <int MODE>
__global__ void __launch_bounds__(kOThreads, 1)
    k_oproj(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
            const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmX,
            const __grid_constant__ CUtensorMap tmY, const OParams p) {
  const int ntile = tiles_of_cta<MODE>(p);
  if (ntile == 0) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  OCtl& C = *reinterpret_cast<OCtl*>(base + kOData);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &C.abort;
  const int ksteps = p.K / 64;
  auto A = [&](int s) { return base + kOffA + s * kABytes; };
  auto A2 = [&](int s) { return base + kOffA2 + s * kABytes; };
  auto B = [&](int s) { return base + (MODE == kDrift ? kOffB2 : kOffB) + s * kBBytes; };
  uint8_t* X = base + kOffX;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kOStages; ++s) {
      mbar_init(&C.full[s], 1);
      mbar_init(&C.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&C.acc_full[b], 1);
      mbar_init(&C.acc_empty[b], 4);
    }
    mbar_init(&C.x_full, 1);
    C.abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
    if (MODE == kDrift) prefetch_tensormap(&tmA2);
    if (MODE == kResidual) {
      prefetch_tensormap(&tmY);
      if (p.has_x) prefetch_tensormap(&tmX);
    }
  }
  if (warp == 1) tmem_alloc(&C.tmem_base, kOCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = C.tmem_base;

  if (warp == 0) {
    // ================================ loads ==========================================
    const uint32_t bytes = (MODE == kDrift ? 2 * kABytes : kABytes) + kBBytes;
    int it = 0;
    bool failed = false;
    for (int k = 0; k < ntile && !failed; ++k) {
      int mt, nt;
      tile_coords<MODE>(p, k, mt, nt);
      for (int ks = 0; ks < ksteps; ++ks, ++it) {
        const int s = it % kOStages, u = it / kOStages;
        if (u > 0 && !o_wait(&C.empty[s], (u - 1) & 1, abort)) {
          failed = true;
          break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&C.full[s], bytes);
          tma_load_3d(A(s), &tmA, &C.full[s], 64 * ks, kOM * mt, 0);
          if (MODE == kDrift) tma_load_3d(A2(s), &tmA2, &C.full[s], 64 * ks, kOM * mt, 0);
          tma_load_3d(B(s), &tmB, &C.full[s], 64 * ks, kON * nt, 0);
        }
        __syncwarp();
      }
    }
    if (failed && lane == 0) {
      o_give_up(C, p.status);
      volatile int no_abort = 0;  // copies already issued land before the memory goes away
      for (int q = max(0, it - kOStages); q < it; ++q)
        mbar_wait(&C.full[q % kOStages], (q / kOStages) & 1, &no_abort, kODrainNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ================================ MMAs ===========================================
    const bool leader = elect_one();
    const uint32_t idesc = idesc_bf16_f32(kOM, kON, false);
    int it = 0;
    bool failed = false;
    if (__popc(__ballot_sync(0xffffffffu, leader)) != 1) {  // exactly one issuing lane
      if (lane == 0) {
        flag_status(p.status, kStatusBadRow);
        *abort = 1;
      }
      failed = true;
    }
    for (int k = 0; k < ntile && !failed; ++k) {
      const int b = MODE == kDrift ? 0 : (k & 1);
      const int use = MODE == kDrift ? k : (k >> 1);  // earlier uses of accumulator b
      if (use > 0 && !o_wait(&C.acc_empty[b], (use - 1) & 1, abort)) {
        failed = true;
        break;
      }
      tc_fence_after();
      const uint32_t acc = tmem + (MODE == kDrift ? 0u : (uint32_t)kON * b);
      for (int ks = 0; ks < ksteps; ++ks, ++it) {
        const int s = it % kOStages;
        if (!o_wait(&C.full[s], (it / kOStages) & 1, abort)) {
          failed = true;
          break;
        }
        tc_fence_after();
        if (leader) {
          const uint32_t a = smem_u32(A(s)), bb = smem_u32(B(s));
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_bf16_ss(acc, sdesc_sw128(a + 32 * kk), sdesc_sw128(bb + 32 * kk), idesc,
                        (ks > 0 || kk > 0) ? 1u : 0u);
          if (MODE == kDrift) {
            const uint32_t a2 = smem_u32(A2(s));
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16_ss(tmem + kON, sdesc_sw128(a2 + 32 * kk), sdesc_sw128(bb + 32 * kk), idesc,
                          (ks > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(&C.empty[s]);
          if (ks + 1 == ksteps) mma_commit(&C.acc_full[b]);
        }
        __syncwarp();
      }
    }
    if (failed && lane == 0) {
      o_give_up(C, p.status);
      if (it > 0) {  // MMAs still running must finish before TMEM is freed
        volatile int no_abort = 0;
        const int q = it - 1;
        mbar_wait(&C.empty[q % kOStages], (q / kOStages) & 1, &no_abort, kODrainNs);
      }
    }
    __syncwarp();
  } else {
    // ================================ epilogue =======================================
    const int quarter = warp & 3;
    const int r = 32 * quarter + lane;  // row of the tile = TMEM lane
    const uint32_t lane_base = (uint32_t)(32 * quarter) << 16;
    const bool leader = (warp == 2 && lane == 0);
    float rowsum = 0.f;
    if (MODE == kResidual && p.has_x && leader) {  // the first tile's x
      int mt, nt;
      tile_coords<MODE>(p, 0, mt, nt);
      mbar_arrive_expect_tx(&C.x_full, 4 * 16384);
#pragma unroll
      for (int q = 0; q < 4; ++q) tma_load_3d(X + q * 16384, &tmX, &C.x_full, kON * nt + 64 * q, kOM * mt, 0);
    }
    for (int k = 0; k < ntile; ++k) {
      int mt, nt;
      tile_coords<MODE>(p, k, mt, nt);
      const int b = MODE == kDrift ? 0 : (k & 1);
      const int use = MODE == kDrift ? k : (k >> 1);
      bool ok = o_wait(&C.acc_full[b], use & 1, abort);
      if (MODE == kResidual && p.has_x && ok) ok = o_wait(&C.x_full, k & 1, abort);
      if (!o_epi_sync_and(ok)) {  // the four warps leave together
        if (!ok && lane == 0) o_give_up(C, p.status);
        break;
      }
      tc_fence_after();
      if (MODE == kDrift) {
#pragma unroll 1
        for (int q = 0; q < kON / 32; ++q) {
          uint32_t va[32], vb[32];
          RESS_TMEM_LD32(tmem + lane_base + 32 * q, va);
          RESS_TMEM_LD32(tmem + kON + lane_base + 32 * q, vb);
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float d = __uint_as_float(va[e]) - __uint_as_float(vb[e]);
            rowsum = fmaf(d, d, rowsum);
          }
        }
      } else {
        const uint32_t acc = tmem + (uint32_t)kON * b + lane_base;
#pragma unroll 1
        for (int q = 0; q < kON / 32; ++q) {  // channels 32q .. 32q + 31: box q/2, chunks 4(q%2)..
          uint32_t v[32];
          RESS_TMEM_LD32(acc + 32 * q, v);
          uint8_t* row = X + (q >> 1) * 16384 + r * 128;
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            uint4* at = reinterpret_cast<uint4*>(row + (((4 * (q & 1) + c) ^ (r & 7)) << 4));
            uint4 xv = make_uint4(0u, 0u, 0u, 0u);
            if (p.has_x) xv = *at;
            const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
            uint32_t yw[4];
#pragma unroll
            for (int e = 0; e < 4; ++e)
              yw[e] = cvt_bf16x2(__uint_as_float(v[8 * c + 2 * e]) + bf16_lo(xw[e]),
                                 __uint_as_float(v[8 * c + 2 * e + 1]) + bf16_hi(xw[e]));
            *at = make_uint4(yw[0], yw[1], yw[2], yw[3]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&C.acc_empty[b]);  // the accumulator may be reused
      if (MODE == kResidual) {
        fence_proxy_async_smem();
        o_epi_sync();
        if (leader) {
#pragma unroll 1
          for (int q = 0; q < 4; ++q)
            if (kON * nt + 64 * q < p.Dm) tma_store_3d(&tmY, X + q * 16384, kON * nt + 64 * q, kOM * mt, 0);
          bulk_commit();
          bulk_wait_read_all();  // the staging area is free again
          if (p.has_x && k + 1 < ntile) {
            int mt2, nt2;
            tile_coords<MODE>(p, k + 1, mt2, nt2);
            mbar_arrive_expect_tx(&C.x_full, 4 * 16384);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              tma_load_3d(X + q * 16384, &tmX, &C.x_full, kON * nt2 + 64 * q, kOM * mt2, 0);
          }
        }
      }
    }
    if (MODE == kDrift) {
      C.rowsum[r] = rowsum;
      o_epi_sync();
      if (threadIdx.x - 64 < 2) {  // one thread per 64-token block of the stripe, rows in order
        const int blk = 2 * blockIdx.x + (threadIdx.x - 64);
        if (blk < p.nb && !*abort) {
          float s = 0.f;
          for (int q = 0; q < 64; ++q) s += C.rowsum[64 * (threadIdx.x - 64) + q];
          p.drift[blk] = s;
        }
      }
    }
    if (leader) bulk_wait_read_all();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kOCols);
  }
}

// A row-major bf16 matrix [rows, cols] as a 3-D tensor {cols, rows, 1}; box {64, box_rows, 1},
// 128-byte swizzle.  Loads past the edges read zeros; stores past them are dropped.
bool make_bf16_map(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, 1};
  cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)rows * cols * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count_of_device() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

template <int MODE>
cudaError_t launch_oproj_impl(const OProjArgs& a, cudaStream_t st) {
  const int K = a.H * 64;
  CUtensorMap ta, ta2, tb, tx, ty;
  if (!make_bf16_map(&ta, a.O, a.N, K, kOM) || !make_bf16_map(&tb, a.W_o, a.Dm, K, kON))
    return cudaErrorInvalidValue;
  ta2 = ta;
  tx = ta;
  ty = ta;
  if (MODE == kDrift && !make_bf16_map(&ta2, a.O2, a.N, K, kOM)) return cudaErrorInvalidValue;
  if (MODE == kResidual) {
    if (!make_bf16_map(&ty, a.y, a.N, a.Dm, kOM)) return cudaErrorInvalidValue;
    if (a.x && !make_bf16_map(&tx, a.x, a.N, a.Dm, kOM)) return cudaErrorInvalidValue;
  }
  OParams p;
  p.N = a.N;
  p.K = K;
  p.Dm = a.Dm;
  p.nb = (a.N + 63) / 64;
  p.mtiles = (a.N + kOM - 1) / kOM;
  p.ntiles = (a.Dm + kON - 1) / kON;
  p.has_x = a.x != nullptr;
  p.drift = a.drift;
  p.status = a.status;
  const size_t smem = kOData + sizeof(OCtl) + 1024;
  cudaError_t e = cudaFuncSetAttribute(k_oproj<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int grid = MODE == kDrift ? p.mtiles : min(p.mtiles * p.ntiles, sm_count_of_device());
  k_oproj<MODE><<<grid, kOThreads, smem, st>>>(ta, ta2, tb, tx, ty, p);
  note_launch();
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_out_proj(const OProjArgs& a, cudaStream_t st) {
  return launch_oproj_impl<kResidual>(a, st);
}

cudaError_t launch_token_drift(const OProjArgs& a, cudaStream_t st) {
  return launch_oproj_impl<kDrift>(a, st);
}

}  // namespace ress
