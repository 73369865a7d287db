// The row-by-block inner products of the selection on the tensor cores.  For one head and
// every candidate row i and block j, with x_i a per-row 64-vector and w_j a per-block one:
//   logits (Sec. 4.1):        L_ij = q_bar_i . k_bar_j / sqrt(64) * log2(e)  (j < nb)
//   drift norms (Eq. 9):      q_ij = ||y~_i||^2 + ||z~_j||^2 - 2 y~_i . z~_j   (j < nb)
//   round gains (Eq. 14/15):  t_ij = c_i - g~_i . z~_j,  c_i = y~_i . g~_i     (j < |P|)
// The rows P (as logits), q or t of the workspace receive the results.  The logits are kept
// in base-2 units, so that P_ij = 2^(L_ij - m_i) / Z_i; each 128-block slice of a row also
// yields its max and its sum of 2^(L - max), from which k_yagg assembles the softmax of the
// row (the pooled map P).
//
// Both operands are fp32; each is held as the sum of three bf16 terms (hi + mid + lo,
// written by the kernels that produce the vectors), and the product is accumulated in fp32
// TMEM from the six term products whose size is at least 2^-16 of hi.hi:
//   mid.mid + hi.lo + lo.hi + hi.mid + mid.hi + hi.hi      (smallest first)
// The three dropped products are below 2^-23 of |x||w| together, the size of the fp32
// rounding of the dot product itself.
//
// One CTA per 128 x 128 tile of (i, j) of one head, 128 threads:
//   thread 0   TMA of the six 128 x 64 bf16 term tiles (128-byte swizzle) on one mbarrier;
//   warp 0     converged MMA warp, one elected lane issues 6 x 4 tcgen05.mma M128 N128 K16
//              (A = x terms, B = w terms, both K-major from shared memory) and commits;
//   warps 0-3  epilogue: tcgen05.ld of the accumulator rows (warp w: rows 32w..32w+31),
//              the result into shared memory (the operand tiles are free by then) as four
//              32-column boxes in the 128-byte-swizzled layout, which thread 0 writes out
//              with TMA bulk tensor stores (rows past nb and columns past the row stride
//              are clipped by the copy; rows past |P| are never read).
// Every mbarrier wait is bounded; a wait that gives up records RESS_ETIMEOUT, lets copies
// and MMAs already issued finish (again bounded), frees TMEM and returns.

#include <cudaTypedefs.h>

#include "ress_internal.cuh"
#include "sm100_ptx.cuh"

namespace ress {
using namespace ptx;

namespace {

constexpr int kDotThreads = 128;
constexpr int kDotTile = 128;                     // rows i and blocks j per CTA
constexpr uint32_t kTermBytes = kDotTile * 128;   // 128 x 64 bf16
constexpr uint32_t kDotCols = 128;                // TMEM columns: one fp32 128 x 128 tile
constexpr uint64_t kDotWaitNs = 2000000000ull;    // 2 s per wait
constexpr uint64_t kDotDrainNs = 200000000ull;    // 0.2 s to drain after an abort

enum DotMode { kDotGain = 0, kDotLogit = 1, kDotDist = 2 };
constexpr float kLogitScale = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)

struct __align__(1024) DotSmem {
  uint8_t A[3][kTermBytes];  // row-vector terms (hi, mid, lo) of rows i0 .. i0 + 127
  uint8_t B[3][kTermBytes];  // block-vector terms of blocks j0 .. j0 + 127
  float bcol[kDotTile];      // drift norms: ||z~_j||^2 of the tile's blocks
  uint64_t full, done;
  uint32_t tmem_base;
  int abort;
};

struct DotParams {
  int nb, ncand, round;  // key blocks (columns), candidate key blocks
  int nq, nqc;           // query blocks (rows), candidate query blocks
  float rho;
  const float* a;     // per row: c_i (gains) or ||y~_i||^2 (drift norms), [H, nb]
  const float* b;     // per block: ||z~_j||^2 (drift norms), [H, nb]
  float2* lstat;      // logits: per row and 128-block slice (max, sum 2^(L - max))
  int nslices;        // ceil(nb / 128)
  int ld;             // row stride of the output
  uint32_t* status;
  Budgets bud;
};

// (A term, B term) of product q of the six, smallest first: 4 bits per q.
constexpr uint32_t kTermA = 0x010201u;  // q = 0..5 -> 1, 0, 2, 0, 1, 0
constexpr uint32_t kTermB = 0x001021u;  // q = 0..5 -> 1, 2, 0, 1, 0, 0

// Bounded wait by a whole warp (all lanes test once; otherwise lane 0 polls and broadcasts).
__device__ __forceinline__ bool dot_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                         uint64_t limit_ns) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, limit_ns) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

template <int MODE>
__global__ void __launch_bounds__(kDotThreads)
    k_dot(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
          const __grid_constant__ CUtensorMap tmOut, const DotParams p) {
  const int h = blockIdx.z, i0 = blockIdx.y * kDotTile, j0 = blockIdx.x * kDotTile;
  if (MODE == kDotGain && swap_count(p.bud.c[h], p.ncand, p.round, p.rho) <= 0) return;
  extern __shared__ uint8_t smem_raw[];
  DotSmem& S = *reinterpret_cast<DotSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;

  if (threadIdx.x == 0) {
    mbar_init(&S.full, 1);
    mbar_init(&S.done, 1);
    S.abort = 0;
    fence_barrier_init();
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
    prefetch_tensormap(&tmOut);
  }
  if (MODE == kDotDist) {
    const int j = j0 + (int)threadIdx.x;  // kDotThreads == kDotTile
    S.bcol[threadIdx.x] = j < p.nb ? p.b[(int64_t)h * p.nb + j] : 0.f;
  }
  if (warp == 0) tmem_alloc(&S.tmem_base, kDotCols);
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
        tma_load_4d(S.A[s], &tmA, &S.full, 0, i0, h, s);
        tma_load_4d(S.B[s], &tmB, &S.full, 0, j0, h, s);
      }
    }
    __syncwarp();
    const bool leader = elect_one();
    if (__popc(__ballot_sync(0xffffffffu, leader)) != 1) {  // exactly one issuing lane
      if (lane == 0) {
        flag_status(p.status, kStatusBadRow);
        *abort = 1;
      }
    } else if (dot_wait(&S.full, 0, abort, kDotWaitNs)) {
      tc_fence_after();
      const uint32_t idesc = idesc_bf16_f32(kDotTile, kDotTile, false);
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
      if (lane == 0) mbar_wait(&S.full, 0, &no_abort, kDotDrainNs);
      __syncwarp();
    }
  }

  // ---- epilogue: warp w holds rows 32w .. 32w + 31 of the tile (TMEM lanes) ----------
  bool ok = dot_wait(&S.done, 0, abort, kDotWaitNs);
  if (!ok && lane == 0 && !*abort) {
    flag_status(p.status, kStatusTimeout);
    *abort = 1;
  }
  if (ok) {
    tc_fence_after();
    const int r = 32 * warp + lane;  // row of the tile = TMEM lane
    const int i = i0 + r;
    const int64_t ri = (int64_t)h * p.nq + i;
    float a = 0.f;
    if (MODE != kDotLogit && i < p.nq) a = p.a[ri];
    float pm = -INFINITY, ps = 0.f;  // logits: running max and sum over the slice
    uint8_t* stage = &S.A[0][0];     // 4 boxes of 128 rows x 32 fp32, 16 KB each
#pragma unroll 1
    for (int q = 0; q < kDotTile / 32; ++q) {
      uint32_t v[32];
      RESS_TMEM_LD32(tmem + ((uint32_t)(32 * warp) << 16) + 32 * q, v);
      float o[32];
      if (MODE == kDotGain) {
#pragma unroll
        for (int k = 0; k < 32; ++k) o[k] = a - __uint_as_float(v[k]);
      } else if (MODE == kDotLogit) {
        const int jq = j0 + 32 * q;
        float cm = -INFINITY;
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          o[k] = __uint_as_float(v[k]) * kLogitScale;
          if (jq + k < p.nb) cm = fmaxf(cm, o[k]);
        }
        if (cm > pm) {
          ps = (pm == -INFINITY) ? 0.f : ps * exp2f(pm - cm);
          pm = cm;
        }
        // the sum in four interleaved partial sums, with the SFU's exp2 (relative error
        // about 2^-22: far below what the row's softmax needs, and half the instructions)
        float sp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int k = 0; k < 32; ++k)
          if (jq + k < p.nb) sp[k & 3] += ex2(o[k] - pm);
        ps += (sp[0] + sp[1]) + (sp[2] + sp[3]);
      } else {
        // ||z~_j||^2 of this quarter's 32 blocks, broadcast from shared memory
        const float4* bq = reinterpret_cast<const float4*>(S.bcol + 32 * q);
#pragma unroll
        for (int k4 = 0; k4 < 8; ++k4) {
          const float4 bz = bq[k4];
          const float b4[4] = {bz.x, bz.y, bz.z, bz.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int k = 4 * k4 + e;
            o[k] = fmaxf(fmaf(-2.0f, __uint_as_float(v[k]), a + b4[e]), 0.f);
          }
        }
      }
      uint8_t* row = stage + q * 16384 + r * 128;
#pragma unroll
      for (int k = 0; k < 8; ++k)  // 16-byte chunk k of the row goes to chunk k ^ (r mod 8)
        *reinterpret_cast<float4*>(row + ((k ^ (r & 7)) << 4)) =
            make_float4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
    }
    if (MODE == kDotLogit && i < p.nqc)
      p.lstat[ri * p.nslices + blockIdx.x] = make_float2(pm, ps);
    fence_proxy_async_smem();
  }
  __syncthreads();
  if (ok && threadIdx.x == 0) {
#pragma unroll 1
    for (int q = 0; q < kDotTile / 32; ++q)
      if (j0 + 32 * q < p.ld) tma_store_3d(&tmOut, &S.A[0][0] + q * 16384, j0 + 32 * q, i0, h);
    bulk_commit();
    bulk_wait_read_all();  // the boxes are read before the shared memory goes away
  }
  if (warp == 0 && issued && !ok) {  // MMAs still running: let them finish before the free
    volatile int no_abort = 0;
    if (lane == 0) mbar_wait(&S.done, 0, &no_abort, kDotDrainNs);
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kDotCols);
  }
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
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

// bf16 [3][H][nb][64] viewed as {64, nb, H, 3}; box {64, rows, 1, 1}, 128-byte swizzle.
// Rows past nb read as zeros.
bool make_term_map(CUtensorMap* m, const void* base, int nb, int H, int rows) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[4] = {64, (cuuint64_t)nb, (cuuint64_t)H, 3};
  cuuint64_t strides[3] = {128, (cuuint64_t)nb * 128, (cuuint64_t)H * nb * 128};
  cuuint32_t box[4] = {64, (cuuint32_t)rows, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp32 [H][nb][ld] viewed as {ld, nb, H}; box {32, 128, 1}, 128-byte swizzle.  Loads past
// the edges read zeros; stores past them are dropped.
bool make_row_map(CUtensorMap* m, void* base, int nb, int H, int ld) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)ld, (cuuint64_t)nb, (cuuint64_t)H};
  cuuint64_t strides[2] = {(cuuint64_t)ld * 4, (cuuint64_t)nb * ld * 4};
  cuuint32_t box[3] = {32, (cuuint32_t)kDotTile, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

template <int MODE>
cudaError_t launch_dot(const SelectArgs& a, int64_t a_terms, int64_t b_terms, int64_t out,
                       const float* rowv, const float* colv, int ncols, int round, float rho,
                       cudaStream_t st) {
  const Shape& s = a.s;
  if (s.ncand <= 0 || s.nqc <= 0) return cudaSuccess;
  CUtensorMap ta, tb, to;
  if (!make_term_map(&ta, a.ws + a_terms, s.nq, s.H, kDotTile) ||
      !make_term_map(&tb, a.ws + b_terms, s.nb, s.H, kDotTile) ||
      !make_row_map(&to, a.ws + out, s.nq, s.H, s.ld))
    return cudaErrorInvalidValue;
  DotParams p;
  p.nb = s.nb;
  p.ncand = s.ncand;
  p.nq = s.nq;
  p.nqc = s.nqc;
  p.round = round;
  p.rho = rho;
  p.a = rowv;
  p.b = colv;
  p.lstat = (float2*)(a.ws + a.L.lstat);
  p.nslices = (s.nb + kDotTile - 1) / kDotTile;
  p.ld = s.ld;
  p.status = (uint32_t*)(a.ws + a.L.status);
  for (int h = 0; h < RESS_MAX_HEADS; ++h) p.bud.c[h] = a.c[h];
  const size_t smem = sizeof(DotSmem) + 1024;
  cudaError_t e =
      cudaFuncSetAttribute(k_dot<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((ncols + kDotTile - 1) / kDotTile, (s.nqc + kDotTile - 1) / kDotTile, s.H);
  k_dot<MODE><<<grid, kDotThreads, smem, st>>>(ta, tb, to, p);
  note_launch();
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gain(const SelectArgs& a, int round, float rho, cudaStream_t st) {
  return launch_dot<kDotGain>(a, a.L.asplit, a.L.zsplit, a.L.t, (const float*)(a.ws + a.L.cdot),
                              nullptr, a.s.ncand, round, rho, st);
}

cudaError_t launch_logits(const SelectArgs& a, cudaStream_t st) {
  return launch_dot<kDotLogit>(a, a.L.asplit, a.L.ksplit, a.L.P, nullptr, nullptr, a.s.nb, 0,
                               0.f, st);
}

cudaError_t launch_drift_norms(const SelectArgs& a, cudaStream_t st) {
  return launch_dot<kDotDist>(a, a.L.asplit, a.L.zsplit, a.L.q, (const float*)(a.ws + a.L.ny),
                              (const float*)(a.ws + a.L.nz), a.s.nb, 0, 0.f, st);
}

}  // namespace ress
