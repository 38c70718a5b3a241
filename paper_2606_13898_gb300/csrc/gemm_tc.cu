// Grouped bf16 GEMM on the 5th-generation tensor cores (tcgen05) for the
// MMDiT block's linear layers (paper Sec. 2.1, the DiT's QKV, output and MLP
// projections): C[r, n] = sum_k A[r, k] * W_g[n, k] + b_g[n]
// with the text rows (group 0) and the packed image rows (group 1) of the
// row space using their own weights. The image row count is read on the
// device, so no host synchronisation is needed between split and block.
//
// Design (one persistent CTA per SM, 192 threads):
//   warp 0     TMA producer: 128x64 A and 256x64 W tiles, 128-byte swizzle,
//              into a 4-stage shared-memory ring (48 KB per stage)
//   warp 1     MMA issuer: tcgen05.mma M=128 N=256 K=16, fp32 accumulator in
//              TMEM, two accumulators (2 x 256 columns) so the epilogue of one
//              tile overlaps the main loop of the next
//   warps 2-5  epilogue: tcgen05.ld 32 columns at a time, bias / GELU /
//              residual add, vector stores
// Every mbarrier wait is bounded; on a timeout the CTA latches an error code
// (read by hilo_sync_status), stops, frees its TMEM and returns.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "gemm_epi.cuh"
#include "internal.h"

namespace hilo {

__device__ int g_gemm_err;

namespace {

constexpr int BM = 128, BK = 64;
constexpr int GEMM_THREADS = 192;

// Tile configuration by tile width: 128x256 tiles with a 4-stage ring, or
// 128x128 tiles with a 6-stage ring (for narrow outputs, N <= 1024).
template <int BN>
struct TileCfg {
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  static constexpr int A_STAGE_BYTES = BM * BK * 2;
  static constexpr int B_STAGE_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EPI_SMEM_BYTES + 1024 + 256;
};

struct GemmParams {
  int N, K;
  uint32_t idesc;
  int row_base[2];
  int rows_static[2];
  const int32_t* rows_dev[2];
  const __nv_bfloat16* bias[2];
  int epilogue;
  void* out;
  const void* resid_src[2];
  int resid_f32;
};

struct Tile {
  int g, m0, n0, rows, row_base;
};

template <int BN>
struct Sched {
  // two row groups, kept in scalars (no runtime-indexed arrays, which would
  // live in local memory)
  int mt0, mt1, rows0, rows1, nt, total;
  __device__ void init(const GemmParams& p) {
    nt = (p.N + BN - 1) / BN;
    // a device row count is bounded by the group's capacity (rows_static)
    rows0 = p.rows_dev[0] ? min(*p.rows_dev[0], p.rows_static[0]) : p.rows_static[0];
    rows1 = p.rows_dev[1] ? min(*p.rows_dev[1], p.rows_static[1]) : p.rows_static[1];
    mt0 = (rows0 + BM - 1) / BM;
    mt1 = (rows1 + BM - 1) / BM;
    total = (mt0 + mt1) * nt;
  }
  __device__ Tile get(const GemmParams& p, int t) const {
    Tile r;
    r.g = t < mt0 * nt ? 0 : 1;
    if (r.g) t -= mt0 * nt;
    const int mtg = r.g ? mt1 : mt0;
    r.row_base = r.g ? p.row_base[1] : p.row_base[0];
    r.m0 = r.row_base + (t % mtg) * BM;
    r.n0 = (t / mtg) * BN;
    r.rows = r.g ? rows1 : rows0;
    return r;
  }
};

template <int BN>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                const __grid_constant__ CUtensorMap tmB1, const __grid_constant__ CUtensorMap tmOut,
                const __grid_constant__ GemmParams p) {
  using Cfg = TileCfg<BN>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr int STAGE_BYTES = Cfg::STAGE_BYTES;
  constexpr int A_STAGE_BYTES = Cfg::A_STAGE_BYTES;
  constexpr uint32_t TMEM_COLS = Cfg::TMEM_COLS;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* epi_stage = smem + STAGES * STAGE_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_stage + EPI_SMEM_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* err = &g_gemm_err;

  pdl_trigger();
  const int warp = warp_id(), lane = lane_id();
  Sched<BN> sc;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 4);  // one arrive per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB0);
    tma_prefetch_desc(&tmB1);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int kblocks = p.K / BK;
  pdl_wait();  // the row counts and A are written by the previous kernel
  sc.init(p);

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_par = 0;  // per stage: armed at least once, parity of the last arming
      bool ok = true;
      for (int t = blockIdx.x; t < sc.total && ok; t += gridDim.x) {
        const Tile tl = sc.get(p, t);
        const CUtensorMap* tb = tl.g ? &tmB1 : &tmB0;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, DEV_TIMEOUT_GEMM)) {
            ok = false;
            break;
          }
          unsigned char* sa = smem + stage * STAGE_BYTES;
          mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
          tma_load_2d(sa, &tmA, &full[stage], kb * BK, tl.m0);
          tma_load_2d(sa + A_STAGE_BYTES, tb, &full[stage], kb * BK, tl.n0);
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // wait (bounded) for the bulk copies already in flight, so that none
        // lands in shared memory after this CTA has exited
        for (int s = 0; s < STAGES; ++s) {
          if (!((armed >> s) & 1u)) continue;
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(smem_u32(&full[s]), (armed_par >> s) & 1u)) {
            if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS / 4) break;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      const uint32_t idesc = p.idesc;
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < sc.total && ok; t += gridDim.x) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, err, DEV_TIMEOUT_GEMM)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, err, DEV_TIMEOUT_GEMM)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t b_base = a_base + A_STAGE_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = sw128_desc(a_base + k * 32, 16, 1024);
            const uint64_t bd = sw128_desc(b_base + k * 32, 16, 1024);
            umma_bf16(d_tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      // every MMA this thread issued has completed before TMEM is freed
      umma_commit(drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(smem_u32(drain), 0u)) {
        if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS) {
          atomicExch(err, DEV_TIMEOUT_GEMM);
          break;
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 -> TMEM lane quarters 2,3,0,1)
    const int q = warp & 3;
    unsigned char* stage = epi_stage + q * EPI_WARP_BYTES;
    int buf = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    if (warp == 2 && lane == 0) tma_prefetch_desc(&tmOut);
    for (int t = blockIdx.x; t < sc.total; t += gridDim.x) {
      const Tile tl = sc.get(p, t);
      const uint4 bpre = epi_bias_preload<BN>(tl.g ? p.bias[1] : p.bias[0], tl.n0, p.N);
      if (!mbar_wait_warp(&tfull[acc], acc_phase, abort_flag, err, DEV_TIMEOUT_GEMM)) break;
      tc_fence_after();
      EpiSlab sl;
      sl.g = tl.g;
      sl.row0 = tl.m0 + q * 32;
      sl.nvalid = min(32, max(0, tl.rows - (tl.m0 - tl.row_base) - q * 32));
      sl.row_base = tl.row_base;
      sl.n0 = tl.n0;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      const int a = acc;
      epilogue_warp<BN>(p, &tmOut, taddr, sl, bpre, EpiScale{}, stage, buf, [&] {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[a]);
      });
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    epilogue_drain();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int BN>
cudaError_t launch_bn(const GemmArgs& a, int num_sms, cudaStream_t st) {
  using Cfg = TileCfg<BN>;
  CUtensorMap tA, tB0, tB1;
  if (!encode_tmap_bf16_2d(&tA, a.A, a.K, a.R, a.K, BK, BM)) return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_2d(&tB0, a.g[0].weight ? a.g[0].weight : a.g[1].weight, a.K, a.N, a.K,
                           BK, BN))
    return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_2d(&tB1, a.g[1].weight ? a.g[1].weight : a.g[0].weight, a.K, a.N, a.K,
                           BK, BN))
    return cudaErrorInvalidValue;
  CUtensorMap tOut;
  if (!encode_epilogue_map(&tOut, a)) return cudaErrorInvalidValue;
  GemmParams p;
  p.N = a.N;
  p.K = a.K;
  p.idesc = idesc_kind_f16(BM, BN, 0, 0, a.op_f16 ? 0 : 1);
  long long upper = 0;
  for (int g = 0; g < 2; ++g) {
    p.row_base[g] = a.g[g].row_base;
    p.rows_static[g] = a.g[g].rows_dev ? a.g[g].rows_cap : a.g[g].rows_static;
    p.rows_dev[g] = a.g[g].rows_dev;
    p.bias[g] = static_cast<const __nv_bfloat16*>(a.g[g].bias);
    upper += (a.g[g].rows_cap + BM - 1) / BM;
  }
  upper *= (a.N + BN - 1) / BN;
  p.epilogue = a.epilogue;
  p.out = a.out;
  p.resid_src[0] = a.resid_src[0];
  p.resid_src[1] = a.resid_src[1];
  p.resid_f32 = a.resid_f32;
  if (upper <= 0) return cudaSuccess;
  const int grid = static_cast<int>(upper < num_sms ? upper : num_sms);
  cudaError_t e = cudaFuncSetAttribute(gemm_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return launch_pdl(gemm_kernel<BN>, dim3(grid), dim3(GEMM_THREADS), Cfg::SMEM_BYTES, st, tA, tB0, tB1,
                    tOut, p);
}

}  // namespace

cudaError_t launch_gemm(const GemmArgs& a, int num_sms, cudaStream_t st) {
  if (a.K % BK != 0 || a.N % 32 != 0) return cudaErrorInvalidValue;
  // CTA pairs with 256x256 tiles where N allows (half the W traffic per SM);
  // else one CTA per tile: 256-wide tiles, or 128-wide where N is so small
  // that 256 would leave SMs idle.
  if (a.fp8) {
    // e4m3 operands run on the pair kernel only
    if (a.N >= 1024 && gemm_pair_supported(a)) return launch_gemm_pair(a, num_sms, st);
    return cudaErrorInvalidValue;
  }
  if (a.N >= 1024 && gemm_pair_supported(a)) return launch_gemm_pair(a, num_sms, st);
  if (a.N <= 1024) return launch_bn<128>(a, num_sms, st);
  return launch_bn<256>(a, num_sms, st);
}

int gemm_take_device_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_gemm_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_gemm_err, &z, sizeof(int));
  return v;
}

}  // namespace hilo
