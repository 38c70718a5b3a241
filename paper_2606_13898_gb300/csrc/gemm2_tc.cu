// Grouped GEMM on CTA pairs (tcgen05 cta_group::2): same computation and
// epilogues as gemm_tc.cu, with 256x256 output tiles per pair of SMs.
//
// Each CTA of a pair loads 128 rows of A and 128 rows of W (half of the
// tile's 256 output columns) into its own shared memory at identical offsets;
// the even CTA issues tcgen05.mma.cta_group::2 with M = 256, N = 256, which
// reads both CTAs' halves. Compared with one SM computing a 128x256 tile,
// each SM stages and feeds half the W bytes per MAC, so the shared-memory
// traffic per MAC drops by a third and the ring can be 6 stages deep.
//
// Per CTA, 192 threads:
//   warp 0     TMA producer: A and W halves; the completion of both CTAs'
//              copies is counted on the even CTA's "full" barrier
//   warp 1     TMEM allocation (both CTAs); MMA issue (even CTA only)
//   warps 2-5  epilogue over this CTA's 128 rows x 256 columns
// "empty" and "accumulator ready" barriers are signalled in both CTAs by a
// multicast commit; "accumulator free" collects 8 arrivals (4 epilogue warps
// x 2 CTAs) in the even CTA. Every wait is bounded.
//
// FP8 (e4m3 A and W, kind::f8f6f4): a k-block is the same 128-byte swizzled
// row of shared memory holding 128 elements instead of 64, and each MMA
// consumes 32 of them; the epilogue multiplies each accumulator by its row's
// A scale and its column's W scale before the bias.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "gemm_epi.cuh"
#include "internal.h"

namespace hilo {

__device__ int g_gemm2_err;

namespace {

constexpr int PM = 256;   // rows per pair tile (128 per CTA)
constexpr int PN = 256;   // columns per pair tile (128 of W rows staged per CTA)
constexpr int BK = 64;
constexpr int STAGES = 6;
constexpr int HALF_BYTES = 128 * BK * 2;    // 16 KB: one CTA's A or W slice
constexpr int STAGE_BYTES = 2 * HALF_BYTES; // A + W slices of this CTA
constexpr int THREADS = 192;
constexpr uint32_t TMEM_COLS = 512;         // two 128 x 256 fp32 accumulators
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EPI_SMEM_BYTES + 1024 + 256;
constexpr int SPLIT_MIN_KB = 32;            // shortest piece of a tile cut into equal K pieces
constexpr int SPLIT_MAX = 8;                // most equal pieces per tile
constexpr int STREAM_MIN_KB = 16;           // shortest stream-K range

struct Params {
  int N, K;
  uint32_t idesc;
  const float* a_scale;     // FP8: dequantisation scale per row of A (row space)
  const float* b_scale[2];  // FP8: per output column, per weight group
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

struct Sched {
  // two row groups, kept in scalars (no runtime-indexed arrays, which would
  // live in local memory)
  int mt0, mt1, rows0, rows1, nt, total;
  __device__ void init(const Params& p) {
    nt = (p.N + PN - 1) / PN;
    // a device row count is bounded by the group's capacity (rows_static)
    rows0 = p.rows_dev[0] ? min(*p.rows_dev[0], p.rows_static[0]) : p.rows_static[0];
    rows1 = p.rows_dev[1] ? min(*p.rows_dev[1], p.rows_static[1]) : p.rows_static[1];
    mt0 = (rows0 + PM - 1) / PM;
    mt1 = (rows1 + PM - 1) / PM;
    total = (mt0 + mt1) * nt;
  }
  __device__ Tile get(const Params& p, int t) const {
    Tile r;
    r.g = t < mt0 * nt ? 0 : 1;
    if (r.g) t -= mt0 * nt;
    const int mtg = r.g ? mt1 : mt0;
    r.row_base = r.g ? p.row_base[1] : p.row_base[0];
    r.m0 = r.row_base + (t % mtg) * PM;
    r.n0 = (t / mtg) * PN;
    r.rows = r.g ? rows1 : rows0;
    return r;
  }
};

// One unit of a pair's work: k-blocks [k0, k1) of tile t.
struct Work {
  int t, k0, k1;
};

// Pieces per tile of the partial round: the count that makes the longest
// pair's share of the round (rounds of pieces x piece length, in k-blocks)
// shortest, with pieces of at least SPLIT_MIN_KB k-blocks, so that a piece's
// main loop still hides the reduce-add epilogue of the piece before it. Ties
// go to fewer pieces.
__device__ __forceinline__ int tail_splits(int rem, int ncl, int kb) {
  if (rem == 0) return 1;
  int best = 1, cost = kb;  // rem < ncl: one round of whole tiles
  for (int s = 2; s <= SPLIT_MAX && kb / s >= SPLIT_MIN_KB; ++s) {
    const int c = ((rem * s + ncl - 1) / ncl) * ((kb + s - 1) / s);
    if (c < cost) {
      best = s;
      cost = c;
    }
  }
  return best;
}

// The work of pair `cid` of `ncl`. Tiles are dealt round-robin, whole, while
// a full round remains. When the output is accumulated in place (fp32 +=,
// written by TMA reduce-add) the tiles of the last, partial round are cut
// along K instead; each piece adds its partial sum to the output, and only
// the piece that starts at k = 0 adds the bias. Two cuts:
//  * equal pieces (tail_splits of them per tile, when that shortens the
//    round), dealt round-robin piece-major: the pieces that run at the same
//    time cover one or two K ranges, so the pairs share those slices of A
//    and W in L2 even when A and W together exceed it;
//  * otherwise stream-K: the round's k-blocks in equal contiguous ranges of
//    at least STREAM_MIN_KB, one per pair, each spanning one or two tiles
//    (shorter than whole pieces, but every pair at its own K offset).
// Other epilogues deal every tile whole. All roles of the pair walk the same
// sequence.
struct WorkIter {
  int t, t_end, ncl, kb, rem, nsplit, u, u_end;
  long long lo, hi;  // stream-K: this pair's k-block range, over the whole tile sequence
  __device__ WorkIter(const Sched& sc, int cid, int ncl_, int kblocks, bool split) {
    ncl = ncl_;
    kb = kblocks;
    rem = split && sc.total > ncl ? sc.total % ncl : 0;
    t_end = sc.total - rem;
    t = cid;
    nsplit = tail_splits(rem, ncl, kblocks);
    u = cid;
    u_end = nsplit > 1 ? rem * nsplit : 0;
    lo = hi = 0;
    if (rem > 0 && nsplit == 1) {
      const long long w = static_cast<long long>(rem) * kblocks;
      const int np = static_cast<int>(max(1LL, min(static_cast<long long>(ncl), w / STREAM_MIN_KB)));
      if (cid < np) {
        lo = w * cid / np;
        hi = w * (cid + 1) / np;
      }
      lo += static_cast<long long>(t_end) * kblocks;
      hi += static_cast<long long>(t_end) * kblocks;
    }
  }
  __device__ bool next(Work& w) {
    if (t < t_end) {
      w.t = t;
      w.k0 = 0;
      w.k1 = kb;
      t += ncl;
      return true;
    }
    if (u < u_end) {
      const int s = u / rem;  // piece index: u_end > 0 implies rem > 0
      w.t = t_end + (u - s * rem);
      w.k0 = s * kb / nsplit;
      w.k1 = (s + 1) * kb / nsplit;
      u += ncl;
      return true;
    }
    if (lo >= hi) return false;
    w.t = static_cast<int>(lo / kb);
    w.k0 = static_cast<int>(lo % kb);
    const long long end = min(hi, static_cast<long long>(w.t + 1) * kb);
    w.k1 = w.k0 + static_cast<int>(end - lo);
    lo = end;
    return true;
  }
};

template <bool FP8>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    gemm2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                 const __grid_constant__ CUtensorMap tmB1, const __grid_constant__ CUtensorMap tmOut,
                 const __grid_constant__ Params p) {
  // elements per k-block: one 128-byte swizzled row of A / W
  constexpr int BKE = FP8 ? 128 : BK;
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
  int* err = &g_gemm2_err;

  const int warp = warp_id(), lane = lane_id();
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cid = blockIdx.x >> 1;
  const int ncl = gridDim.x >> 1;
  pdl_trigger();
  Sched sc;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 8);  // 4 epilogue warps x 2 CTAs
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
    tmem_alloc_pair(tmem_slot, TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers are initialised before any remote use
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int kblocks = p.K / BKE;
  // The weights do not depend on the previous kernel: while it finishes,
  // pull the first k-blocks of this pair's first weight tile into L2. The
  // tile is exact when it lies in a group whose row count is static (the
  // text rows); in the image rows, whose count is read only after the wait,
  // the column block is a guess, and a wrong one costs only the prefetch.
  if (warp == 0 && lane == 0) {
    const int nt = p.N / PN;
    const int mt0 = p.rows_dev[0] ? 0 : (p.rows_static[0] + PM - 1) / PM;
    const CUtensorMap* tb;
    int n;
    if (cid < mt0 * nt) {
      tb = &tmB0;
      n = cid / mt0;
    } else {
      tb = &tmB1;
      n = (cid - mt0 * nt) % nt;
    }
    const int y = n * PN + 128 * static_cast<int>(rank);
    for (int kb = 0; kb < min(kblocks, STAGES); ++kb) tma_prefetch_l2_2d(tb, kb * BKE, y);
  }
  pdl_wait();  // the row counts and A are written by the previous kernel
  sc.init(p);
  const bool split_k = p.epilogue == EPI_BIAS_RESID_F32;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs)
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_par = 0;  // per stage: armed at least once, parity of the last arming
      bool ok = true;
      WorkIter it(sc, cid, ncl, kblocks, split_k);
      Work w;
      while (ok && it.next(w)) {
        const Tile tl = sc.get(p, w.t);
        const CUtensorMap* tb = tl.g ? &tmB1 : &tmB0;
        for (int kb = w.k0; kb < w.k1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err, DEV_TIMEOUT_GEMM + 256 * 1)) {
            ok = false;
            break;
          }
          unsigned char* sa = smem + stage * STAGE_BYTES;
          const uint32_t full_cl = mapa_shared(smem_u32(&full[stage]), 0);
          if (leader) mbar_arrive_expect_tx(&full[stage], 2 * STAGE_BYTES);
          tma_load_2d_pair(sa, &tmA, full_cl, kb * BKE, tl.m0 + 128 * static_cast<int>(rank));
          tma_load_2d_pair(sa + HALF_BYTES, tb, full_cl, kb * BKE, tl.n0 + 128 * static_cast<int>(rank));
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // let the bulk copies already issued land before the CTA can exit
        const uint64_t t0 = globaltimer_ns();
        if (leader) {
          for (int s = 0; s < STAGES; ++s) {
            if (!((armed >> s) & 1u)) continue;
            while (!mbar_try_wait(smem_u32(&full[s]), (armed_par >> s) & 1u) &&
                   globaltimer_ns() - t0 < HILO_WAIT_LIMIT_NS / 4) {
            }
          }
        } else {
          while (globaltimer_ns() - t0 < 50000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------- MMA issuer (even CTA)
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      WorkIter it(sc, cid, ncl, kblocks, split_k);
      Work w;
      while (ok && it.next(w)) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, err, DEV_TIMEOUT_GEMM + 256 * 2)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * PN);
        for (int kb = w.k0; kb < w.k1; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, err, DEV_TIMEOUT_GEMM + 256 * 3)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t b_base = a_base + HALF_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = sw128_desc(a_base + k * 32, 16, 1024);
            const uint64_t bd = sw128_desc(b_base + k * 32, 16, 1024);
            if (FP8)
              umma_f8_pair(d_tmem, ad, bd, p.idesc, (kb > w.k0 || k > 0) ? 1u : 0u);
            else
              umma_f16_pair(d_tmem, ad, bd, p.idesc, (kb > w.k0 || k > 0) ? 1u : 0u);
          }
          umma_commit_pair(&empty[stage], 0x3);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_pair(&tfull[acc], 0x3);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      umma_commit_pair(drain, 0x1);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(smem_u32(drain), 0u)) {
        if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS) {
          atomicExch(err, DEV_TIMEOUT_GEMM + 256 * 4);
          break;
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 -> TMEM lane quarters 2,3,0,1), both CTAs
    const int q = warp & 3;
    unsigned char* stage = epi_stage + q * EPI_WARP_BYTES;
    int buf = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    if (warp == 2 && lane == 0) tma_prefetch_desc(&tmOut);
    WorkIter it(sc, cid, ncl, kblocks, split_k);
    Work w;
    while (it.next(w)) {
      const Tile tl = sc.get(p, w.t);
      // the bias is added once per tile, by the piece that starts at k = 0
      const uint4 bpre = w.k0 == 0 ? epi_bias_preload<PN>(tl.g ? p.bias[1] : p.bias[0], tl.n0, p.N)
                                   : make_uint4(0u, 0u, 0u, 0u);
      EpiScale escale;
      if (FP8) escale = epi_scale_preload<PN>(p.a_scale, tl.g ? p.b_scale[1] : p.b_scale[0],
                                              tl.m0 + 128 * static_cast<int>(rank) + q * 32,
                                              min(32, max(0, tl.rows - (tl.m0 - tl.row_base) -
                                                                 (128 * static_cast<int>(rank) + q * 32))),
                                              tl.n0, p.N);
      const int off = 128 * static_cast<int>(rank) + q * 32;  // slab offset in the pair tile
      const int nvalid = min(32, max(0, tl.rows - (tl.m0 - tl.row_base) - off));
      if (p.epilogue == EPI_BIAS_RESIDIN_F32 && lane < nvalid && tl.n0 < p.N) {
        // this lane's residual row into L2 while the accumulator is still
        // being computed, so that the epilogue's chunk loads do not each
        // wait for DRAM
        const int esz = p.resid_f32 ? 4 : 2;
        const char* r = static_cast<const char*>(tl.g ? p.resid_src[1] : p.resid_src[0]) +
                        (static_cast<long long>(tl.m0 + off + lane - tl.row_base) * p.N + tl.n0) * esz;
        for (int j = 0; j < PN * esz / 128; ++j) prefetch_l2(r + 128 * j);
      }
      if (!mbar_wait_warp(&tfull[acc], acc_phase, abort_flag, err, DEV_TIMEOUT_GEMM + 256 * 5)) break;
      tc_fence_after();
      EpiSlab sl;
      sl.g = tl.g;
      sl.row0 = tl.m0 + off;
      sl.nvalid = nvalid;
      sl.row_base = tl.row_base;
      sl.n0 = tl.n0;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * PN);
      const int a = acc;
      epilogue_warp<PN>(p, &tmOut, taddr, sl, bpre, escale, stage, buf, [&] {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[a]), 0));
      });
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    epilogue_drain();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no remote arrivals / copies into the peer after this point
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, TMEM_COLS);
  }
}

}  // namespace

bool gemm_pair_supported(const GemmArgs& a) { return a.K % (a.fp8 ? 128 : BK) == 0 && a.N % PN == 0; }

cudaError_t launch_gemm_pair(const GemmArgs& a, int num_sms, cudaStream_t st) {
  if (!gemm_pair_supported(a)) return cudaErrorInvalidValue;
  CUtensorMap tA, tB0, tB1;
  // FP8: bytes are the elements, 128 per swizzled row (box 128 x 128)
  const TmapType tt = a.fp8 ? TMAP_U8 : TMAP_BF16;
  const uint32_t bk = a.fp8 ? 128 : BK;
  if (!encode_tmap_2d(&tA, tt, a.A, a.K, a.R, a.K, bk, 128)) return cudaErrorInvalidValue;
  if (!encode_tmap_2d(&tB0, tt, a.g[0].weight ? a.g[0].weight : a.g[1].weight, a.K, a.N, a.K, bk, 128))
    return cudaErrorInvalidValue;
  if (!encode_tmap_2d(&tB1, tt, a.g[1].weight ? a.g[1].weight : a.g[0].weight, a.K, a.N, a.K, bk, 128))
    return cudaErrorInvalidValue;
  CUtensorMap tOut;
  if (!encode_epilogue_map(&tOut, a)) return cudaErrorInvalidValue;
  Params p;
  p.N = a.N;
  p.K = a.K;
  // format code 0: fp16 for kind::f16, E4M3 for kind::f8f6f4
  p.idesc = idesc_kind_f16(PM, PN, 0, 0, (a.op_f16 || a.fp8) ? 0 : 1);
  p.a_scale = a.a_scale;
  p.b_scale[0] = a.g[0].w_scale;
  p.b_scale[1] = a.g[1].w_scale;
  long long upper = 0;
  for (int g = 0; g < 2; ++g) {
    p.row_base[g] = a.g[g].row_base;
    p.rows_static[g] = a.g[g].rows_dev ? a.g[g].rows_cap : a.g[g].rows_static;
    p.rows_dev[g] = a.g[g].rows_dev;
    p.bias[g] = static_cast<const __nv_bfloat16*>(a.g[g].bias);
    upper += (a.g[g].rows_cap + PM - 1) / PM;
  }
  upper *= a.N / PN;
  p.epilogue = a.epilogue;
  p.out = a.out;
  p.resid_src[0] = a.resid_src[0];
  p.resid_src[1] = a.resid_src[1];
  p.resid_f32 = a.resid_f32;
  if (upper <= 0) return cudaSuccess;
  auto* kern = a.fp8 ? gemm2_kernel<true> : gemm2_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  // persistent grid: as many co-resident CTA pairs as the device holds
  static int max_pairs = 0;
  if (max_pairs == 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (num_sms / 2), 1, 1);
    cfg.blockDim = dim3(THREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 2;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    max_pairs = n;
  }
  const long long pairs = upper < max_pairs ? upper : max_pairs;
  return launch_pdl(kern, dim3(static_cast<int>(2 * pairs)), dim3(THREADS), SMEM_BYTES, st, tA, tB0, tB1, tOut,
                    p);
}

int gemm2_take_device_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_gemm2_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_gemm2_err, &z, sizeof(int));
  return v;
}

}  // namespace hilo
