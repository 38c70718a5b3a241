// Joint variable-length softmax attention of the MMDiT block on tcgen05
// (paper Sec. 2.1: the DiT of the editing generalist; Sec. 2.3: the
// compressed image tokens attend jointly with the text tokens).
//
// Image b attends over its joint sequence [T text rows ; L_b packed image
// rows] (non-causal, scale 1/sqrt(head_dim)); L_b comes from the device
// array cu_img, so the compressed sequence lengths never travel to the host.
// The text rows and the image rows of one image live in two separate ranges
// of the row space; queries and keys/values are tiled per range (128 rows per
// tile, the ragged last tile masked).
//
// A persistent grid, one CTA per SM. The query tiles of all (image, head)
// groups, in image, head, tile order, are cut into one contiguous range per
// CTA (ceil(tiles / CTAs) each), so every CTA has the same work, whatever the
// count of tiles, which only the device knows. A CTA walks its range as jobs:
// two tiles of one group form a pair (one query tile per softmax warpgroup,
// sharing every K/V tile); a lone tile at the edge of the range or of its
// group is a split job, whose key tiles alternate between the warpgroups
// (even tiles to the first, odd to the second); the second warpgroup then
// hands its row maxima and sums to the first, which merges the two
// accumulators (each relative to its own maximum) and writes the rows. At
// the 64x64 workload (456 query tiles on 152 SMs) every CTA runs one pair and
// one split job instead of two pairs on some SMs and one on the others.
// Between jobs, the next job's Q is loaded as soon as the previous job's
// MMAs are done, and its K once the previous output rows (staged in the K
// stages) are out. 384 threads in three warpgroups:
//   warps 0-3    softmax of query tile 0 (one query row per thread)
//   warps 4-7    softmax of query tile 1 (of a split job: the odd key tiles)
//   warp 8       TMA: Q tiles, then K tiles (two stages), 128-byte
//                swizzled boxes of 64 columns
//   warp 10      TMA: V tiles (two stages)
//   warp 9       MMA: S_i = Q_i K^T into TMEM, O_i += P_i V into TMEM. The
//                whole warp walks the schedule and waits, so that stage
//                indices and descriptor words stay warp-uniform; one elected
//                lane issues. (With one lane alone, each MMA's descriptor
//                arithmetic sat on that lane's dependent chain and the issue
//                fell behind the tensor pipe.)
//   warp 11      idle (the third warpgroup gives its registers away)
// Tensor memory holds S_0 | S_1 | O_0 | O_1 (128 columns each). A softmax
// warpgroup reads S_i once into registers and writes the probabilities P_i
// back over the first 64 columns of S_i as packed bf16; the PV product takes
// P_i from tensor memory (A operand) and V from shared memory (MN-major, no
// transpose pass). The two query tiles ping-pong on the tensor core (MMA
// order PV_0(t), S_0(t+1), PV_1(t), S_1(t+1)); S_i(t+1) overwrites P_i(t)
// only after PV_i(t), in issue order. When a softmax warpgroup sees S_i(t),
// every earlier MMA has completed, so O_i may be rescaled and P_i written
// without a further wait. The output accumulators are rescaled only when a
// row's running maximum grows by more than 2^8 (until then the
// probabilities are formed against the older, smaller maximum, so they stay
// <= 256, well inside bf16 range).
// With proportional attention (PROP) every key j carries a weight n_j (the
// number of grid tokens a packed image row stands for; text keys weigh 1):
// softmax(s + ln n) = n e^s / sum(n e^s), so each probability is multiplied
// by its key's weight before the row sum and the bf16 packing, and the row
// maxima (the stabiliser) stay those of the raw logits. Each softmax warp
// fetches the next key tile's 128 weights with asynchronous 4-byte copies
// (zero-filled past the ragged end) into its own double-buffered shared slot
// while it works on the current tile, and reads them back as 16-byte
// broadcasts; no barrier spans warps.
// Every mbarrier wait is bounded (error latched, TMEM freed, CTA returns).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace hilo {

__device__ int g_attn_err;

namespace {

constexpr int BQ = 128;
constexpr int BKV = 128;
// Three warpgroups: two softmax warpgroups and one for TMA, MMA and two idle
// warps. The control warpgroup gives registers to the softmax warpgroups
// (setmaxnreg); launch_hd checks that the shares fit the launch allocation.
constexpr int ATTN_THREADS = 384;
constexpr int PRODUCER_WARP = 8;    // Q and K copies
constexpr int V_PRODUCER_WARP = 10; // V copies
constexpr int MMA_WARP = 9;
constexpr uint32_t SOFTMAX_REGS = 216;
constexpr uint32_t CONTROL_REGS = 72;
constexpr uint32_t ATTN_TMEM_COLS = 512;  // S0 | S1 | O0 | O1
constexpr int BOX_BYTES = 128 * 128;       // 128 rows x 64 16-bit elements
constexpr float RESCALE_LOG2 = 8.0f;

template <int HD, bool PROP>
struct Cfg {
  static constexpr int NBOX = HD / 64;
  static constexpr int TILE_BYTES = NBOX * BOX_BYTES;  // 128 rows x HD
  // Q0 | Q1 | K0 | K1 | V0 | V1
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = 2 * TILE_BYTES;
  static constexpr int OFF_V = 4 * TILE_BYTES;
  static constexpr int DATA_BYTES = 6 * TILE_BYTES;
  // barriers (256 B); with PROP, 8 softmax warps x 2 slots x 128 weights;
  // the row maxima and sums a split job's second warpgroup hands over
  static constexpr int OFF_W = DATA_BYTES + 256;
  static constexpr int OFF_ML = OFF_W + (PROP ? 8 * 2 * BKV * 4 : 0);
  static constexpr int SMEM_BYTES = OFF_ML + 2 * BQ * 4 + 1024;  // + alignment of the base
};

struct AttnParams {
  const int32_t* cu_img;
  const float* n_img;  // PROP: weight of each packed image row
  __nv_bfloat16* out;
  int B, T, heads, d, qt_txt;
  int cap;           // image-row capacity: row offsets are clamped to it
  float scale_log2;  // log2(e) / sqrt(head_dim)
};

// 4-byte asynchronous global -> shared copy; bytes past src_bytes (0 or 4)
// are zero-filled
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Named barrier `id` (1..15) over `nthreads` threads (a multiple of 32).
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Named barrier over `nthreads` threads (a multiple of 32) that also returns
// whether `pred` held for any of them.
__device__ __forceinline__ bool bar_red_or(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(pred ? 1u : 0u), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

// Pairs of fp32 values in one 64-bit register pair: Blackwell's paired fp32
// instructions (fma/mul/add .f32x2) apply the same IEEE operation to both
// halves at one issue slot per pair.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// mbar_wait_warp on two barriers: both phases must complete. The common case
// (both already complete) costs two try_waits and one warp vote.
__device__ __forceinline__ bool mbar_wait2_warp(uint64_t* a, uint32_t pa, uint64_t* b, uint32_t pb,
                                                volatile int* abort, int* err, int code_a, int code_b) {
  bool ok = mbar_try_wait(smem_u32(a), pa) && mbar_try_wait(smem_u32(b), pb);
  if (!ok) ok = mbar_wait(a, pa, abort, err, code_a) && mbar_wait(b, pb, abort, err, code_b);
  return __all_sync(0xffffffffu, ok);
}

// One lane of the warp, the same one for every call with all lanes active.
__device__ __forceinline__ bool elect_one() {
  uint32_t r;
  asm volatile("{\n\t.reg .pred p;\n\telect.sync _|p, 0xffffffff;\n\tselp.u32 %0, 1, 0, p;\n\t}" : "=r"(r));
  return r != 0;
}

// The two 32-bit words of a 128-byte-swizzle shared-memory descriptor: the
// low word holds start address >> 4 (bits 0..13) and LBO >> 4 (bits
// 16..29), the high word SBO >> 4, the descriptor version (bit 46) and the
// swizzle mode (bits 61..63). Shared addresses stay below 2^18 bytes, so
// adding an offset >> 4 to a low word never carries into the LBO field.
__host__ __device__ constexpr uint32_t sw128_lo_lbo(uint32_t lbo) { return ((lbo >> 4) & 0x3FFFu) << 16; }
__host__ __device__ constexpr uint32_t sw128_hi(uint32_t sbo) {
  return ((sbo >> 4) & 0x3FFFu) | (1u << 14) | (2u << 29);
}

// tcgen05.mma kind::f16, A and B from shared memory, descriptors given as words
__device__ __forceinline__ void umma_bf16_w(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo, uint32_t hi,
                                            uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 da, db;\n\t"
      "setp.ne.b32 p, %5, 0;\n\t"
      "mov.b64 da, {%1, %3};\n\t"
      "mov.b64 db, {%2, %3};\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], da, db, %4, p;\n\t}" ::"r"(d_tmem),
      "r"(a_lo), "r"(b_lo), "r"(hi), "r"(idesc), "r"(acc)
      : "memory");
}
// the same with A from tensor memory
__device__ __forceinline__ void umma_bf16_tmem_a_w(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo, uint32_t hi,
                                                   uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 db;\n\t"
      "setp.ne.b32 p, %5, 0;\n\t"
      "mov.b64 db, {%2, %3};\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], db, %4, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "r"(b_lo), "r"(hi), "r"(idesc), "r"(acc)
      : "memory");
}

// The largest of three floats in one instruction (three-input max.f32). A
// maximum is exact, so grouping the row's values by threes gives the same
// result as any other order.
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float y;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
  return y;
}

// Row range of tile j of image b (text tiles first, then image tiles); used
// for both query and key/value tiles.
__device__ __forceinline__ void seq_tile(const AttnParams& p, int b, int L, int j, int& row0,
                                         int& valid) {
  if (j < p.qt_txt) {
    row0 = b * p.T + j * BKV;
    valid = min(BKV, p.T - j * BKV);
  } else {
    const int k = j - p.qt_txt;
    row0 = p.B * p.T + min(p.cu_img[b], p.cap) + k * BKV;
    valid = min(BKV, L - k * BKV);
  }
}

// Packed image rows of image b within the capacity.
__device__ __forceinline__ int img_len(const AttnParams& p, int b) {
  return min(p.cu_img[b + 1], p.cap) - min(p.cu_img[b], p.cap);
}

// Query tiles of all (image, head) groups.
__device__ long long total_qtiles(const AttnParams& p) {
  long long q = 0;
  for (int b = 0; b < p.B; ++b) q += p.qt_txt + (img_len(p, b) + BQ - 1) / BQ;
  return q * p.heads;
}

// A CTA's unit of work: two query tiles of one (image, head) over all key
// tiles (pair), or one query tile whose key tiles are split between the two
// softmax warpgroups -- even tiles to the first, odd tiles to the second --
// and merged at the end (split).
struct Job {
  bool pair;
  int b, h, j0, nkv, L;
};

// The next job of the flat query-tile range [g, end) (tiles ordered by image,
// head, tile): two tiles of one group form a pair, a lone tile at the edge of
// the range or of its group is a split job.
__device__ bool next_job(const AttnParams& p, long long& g, long long end, Job& jb) {
  if (g >= end) return false;
  long long base = 0;
  int b = 0, nq = 0, L = 0;
  for (; b < p.B; ++b) {
    L = img_len(p, b);
    nq = p.qt_txt + (L + BQ - 1) / BQ;
    const long long cnt = static_cast<long long>(nq) * p.heads;
    if (g < base + cnt) break;
    base += cnt;
  }
  if (b >= p.B) return false;
  const long long r = g - base;
  jb.b = b;
  jb.h = static_cast<int>(r / nq);
  jb.j0 = static_cast<int>(r % nq);
  jb.nkv = nq;
  jb.L = L;
  const long long grp_end = base + static_cast<long long>(jb.h + 1) * nq;
  jb.pair = (end < grp_end ? end : grp_end) - g >= 2;
  g += jb.pair ? 2 : 1;
  return true;
}

// Steps of warpgroup i in a job, and the key tile of its step s.
__device__ __forceinline__ int job_steps(const Job& jb, int i) {
  return jb.pair ? jb.nkv : (jb.nkv + 1 - i) / 2;
}
__device__ __forceinline__ int job_tile(const Job& jb, int i, int s) { return jb.pair ? s : 2 * s + i; }

template <int HD, bool PROP>
__global__ void __launch_bounds__(ATTN_THREADS, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm, const __grid_constant__ AttnParams p) {
  using C = Cfg<HD, PROP>;
  pdl_trigger();
  pdl_wait();  // cu_img and q/k/v are written by the previous kernels
  // ---- this CTA's share: a contiguous range of the query tiles of all
  // (image, head) groups, ceil(total / grid) tiles per CTA
  const long long qtiles = total_qtiles(p);
  const long long per = (qtiles + gridDim.x - 1) / gridDim.x;
  const long long g_begin = static_cast<long long>(blockIdx.x) * per;
  const long long g_end = min(qtiles, g_begin + per);
  if (g_begin >= g_end) return;  // uniform across the CTA: nothing allocated yet

  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::DATA_BYTES);
  uint64_t* q_full = bars + 0;
  uint64_t* k_full = bars + 1;    // [2]
  uint64_t* k_empty = bars + 3;   // [2]
  uint64_t* v_full = bars + 5;    // [2]
  uint64_t* v_empty = bars + 7;   // [2]
  uint64_t* s_full = bars + 9;    // [2] per softmax warpgroup
  uint64_t* p_full = bars + 11;   // [2] per softmax warpgroup
  uint64_t* o_done = bars + 13;   // [2] per softmax warpgroup
  uint64_t* drain = bars + 15;
  uint64_t* q_empty = bars + 16;  // every MMA of a job done: Q may be reloaded
  uint64_t* epi_done = bars + 17; // a job's output rows are out: K stages free
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* ml_slot = reinterpret_cast<float*>(smem + C::OFF_ML);  // split merge: m | l of warpgroup 1
  int* err = &g_attn_err;
  auto sQ = [&](int i) { return smem + C::OFF_Q + i * C::TILE_BYTES; };
  auto sK = [&](int st) { return smem + C::OFF_K + st * C::TILE_BYTES; };
  auto sV = [&](int st) { return smem + C::OFF_V + st * C::TILE_BYTES; };

  const int warp = warp_id(), lane = lane_id();
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&o_done[i], 1);
    }
    mbar_init(drain, 1);
    mbar_init(q_empty, 1);
    mbar_init(epi_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == MMA_WARP) {
    tmem_alloc(tmem_slot, ATTN_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // key tile t of a job whose first tile is the CTA's running tile kt0: its
  // stage and the parity of that stage's use
  auto kv_stage = [](uint32_t kt0, int t) { return static_cast<int>((kt0 + t) & 1u); };
  auto kv_phase = [](uint32_t kt0, int t) { return ((kt0 + static_cast<uint32_t>(t)) >> 1) & 1u; };
  if (warp >= 8) {
    // control warpgroup: two TMA producers, the MMA issuer, one idle warp
    setmaxnreg_dec<CONTROL_REGS>();
    if (warp == PRODUCER_WARP || warp == V_PRODUCER_WARP) {
    if (lane == 0) {
      // ---------------- TMA producers: Q and K tiles (warp 8), V tiles
      // (warp 10). Two threads, so that a K copy never queues behind a V
      // stage that is still being read, and the other way round.
      const bool kq = warp == PRODUCER_WARP;
      tma_prefetch_desc(&tm);
      // per stage (bit st): armed at least once, and the parity of the last arming
      uint32_t armed = 0, par = 0;
      bool q_armed = false;
      uint32_t q_par = 0;
      bool ok = true;
      uint32_t kt = 0;
      long long g = g_begin;
      Job jb;
      uint64_t* full = kq ? k_full : v_full;
      uint64_t* empty = kq ? k_empty : v_empty;
      for (uint32_t jn = 0; ok && next_job(p, g, g_end, jb); ++jn) {
        if (kq) {
          // Q of this job once the previous job's MMAs are done with Q
          if (jn > 0 && !mbar_wait(q_empty, (jn - 1) & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 16)) {
            ok = false;
            break;
          }
          int qr0, qv, qr1 = 0, qv1;
          seq_tile(p, jb.b, jb.L, jb.j0, qr0, qv);
          if (jb.pair) seq_tile(p, jb.b, jb.L, jb.j0 + 1, qr1, qv1);
          mbar_arrive_expect_tx(q_full, (jb.pair ? 2 : 1) * C::TILE_BYTES);
#pragma unroll
          for (int j = 0; j < C::NBOX; ++j) {
            tma_load_2d(sQ(0) + j * BOX_BYTES, &tm, q_full, jb.h * HD + 64 * j, qr0);
            if (jb.pair) tma_load_2d(sQ(1) + j * BOX_BYTES, &tm, q_full, jb.h * HD + 64 * j, qr1);
          }
          q_armed = true;
          q_par = jn & 1u;
          // K once the previous job's output rows (staged in the K stages)
          // are out
          if (jn > 0 && !mbar_wait(epi_done, (jn - 1) & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 17)) {
            ok = false;
            break;
          }
        }
        const int col = (kq ? 1 : 2) * p.d + jb.h * HD;
        for (int t = 0; t < jb.nkv; ++t) {
          const int st = kv_stage(kt, t);
          const uint32_t ph = kv_phase(kt, t);
          int row0, valid;
          seq_tile(p, jb.b, jb.L, t, row0, valid);
          if (!mbar_wait(&empty[st], ph ^ 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * (kq ? 1 : 2))) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[st], C::TILE_BYTES);
          unsigned char* dst = kq ? sK(st) : sV(st);
#pragma unroll
          for (int j = 0; j < C::NBOX; ++j) tma_load_2d(dst + j * BOX_BYTES, &tm, &full[st], col + 64 * j, row0);
          armed |= 1u << st;
          par = (par & ~(1u << st)) | (ph << st);
        }
        kt += static_cast<uint32_t>(jb.nkv);
      }
      if (!ok) {
        // wait (bounded) for this thread's bulk copies in flight before the
        // CTA exits
        const uint64_t t0 = globaltimer_ns();
        const uint64_t lim = HILO_WAIT_LIMIT_NS / 4;
        if (q_armed)
          while (!mbar_try_wait(smem_u32(q_full), q_par) && globaltimer_ns() - t0 < lim) {
          }
        for (int st = 0; st < 2; ++st)
          if ((armed >> st) & 1u)
            while (!mbar_try_wait(smem_u32(&full[st]), (par >> st) & 1u) && globaltimer_ns() - t0 < lim) {
            }
      }
    }
  } else if (warp == MMA_WARP) {
    // ---------------- MMA issuer. The whole warp walks the schedule and
    // waits, so that the stage indices and descriptor words stay
    // warp-uniform (no per-MMA moves into the uniform datapath); one elected
    // lane issues the MMAs and commits. Each MMA's shared-memory descriptor
    // is a precomputed high word and a low word that is one add away from
    // its operand's base (start address >> 4 in the low 14 bits, LBO above).
    const bool leader = elect_one();
    constexpr uint32_t idesc_s = idesc_bf16(BQ, BKV, 0, 0);
    constexpr uint32_t idesc_o = idesc_bf16(BQ, HD, 0, 1);
    constexpr uint32_t TILE16 = C::TILE_BYTES >> 4;
    const uint32_t base16 = smem_u32(smem) >> 4;
    const uint32_t q_lo = base16 + (C::OFF_Q >> 4) + sw128_lo_lbo(16);
    const uint32_t k_lo = base16 + (C::OFF_K >> 4) + sw128_lo_lbo(16);
    const uint32_t v_lo = base16 + (C::OFF_V >> 4) + sw128_lo_lbo(BOX_BYTES);
    constexpr uint32_t hi = sw128_hi(1024);
    // S_i = Q_qb K^T (K from stage kst)
    auto issue_s = [&](int i, int qb, int kst) {
      if (leader) {
        const uint32_t a = q_lo + static_cast<uint32_t>(qb) * TILE16, b = k_lo + static_cast<uint32_t>(kst) * TILE16;
#pragma unroll
        for (int k = 0; k < HD / 16; ++k) {
          const uint32_t off = static_cast<uint32_t>((k >> 2) * BOX_BYTES + (k & 3) * 32) >> 4;
          umma_bf16_w(tmem + 128u * i, a + off, b + off, hi, idesc_s, k > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[i]);
      }
      __syncwarp();
    };
    // O_i (+)= P_i V: P_i from the first 64 TMEM columns of S_i (8 columns =
    // 16 keys per MMA), V from stage vst. The last PV_i of a job commits
    // o_done[i] (one phase per job with steps for warpgroup i)
    auto issue_pv = [&](int i, int vst, bool acc, bool last) {
      if (leader) {
        const uint32_t b = v_lo + static_cast<uint32_t>(vst) * TILE16;
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k)
          umma_bf16_tmem_a_w(tmem + 256u + 128u * i, tmem + 128u * i + 8u * k, b + ((k * 2048) >> 4), hi, idesc_o,
                             (acc || k > 0) ? 1u : 0u);
        if (last) umma_commit(&o_done[i]);
      }
      __syncwarp();
    };
    auto commit = [&](uint64_t* bar) {
      if (leader) umma_commit(bar);
      __syncwarp();
    };
    bool ok = true;
    uint32_t kt = 0, sc0 = 0, sc1 = 0;
    long long g = g_begin;
    Job jb;
    for (uint32_t jn = 0; ok && next_job(p, g, g_end, jb); ++jn) {
      const int n0 = job_steps(jb, 0), n1 = job_steps(jb, 1);
      const int qb1 = jb.pair ? 1 : 0;  // the Q buffer of warpgroup 1
      auto wait_k = [&](int t) {
        return mbar_wait_warp(&k_full[kv_stage(kt, t)], kv_phase(kt, t), abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 4);
      };
      auto wait_v = [&](int t) {
        return mbar_wait_warp(&v_full[kv_stage(kt, t)], kv_phase(kt, t), abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 6);
      };
      if (!mbar_wait_warp(q_full, jn & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 3) || !wait_k(0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      // the first S of each warpgroup; a pair shares key tile 0, a split
      // job gives warpgroup 1 key tile 1
      issue_s(0, 0, kv_stage(kt, 0));
      if (jb.pair) {
        issue_s(1, 1, kv_stage(kt, 0));
        commit(&k_empty[kv_stage(kt, 0)]);
      } else {
        commit(&k_empty[kv_stage(kt, 0)]);
        if (n1 > 0) {
          if (!wait_k(1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_s(1, 0, kv_stage(kt, 1));
          commit(&k_empty[kv_stage(kt, 1)]);
        }
      }
      // ping-pong: PV_0(s), S_0(s+1), PV_1(s), S_1(s+1); S_i(s+1)
      // overwrites P_i(s) only after PV_i(s), in issue order
      const int nmax = n0 > n1 ? n0 : n1;
      for (int s = 0; s < nmax && ok; ++s) {
        if (s < n0) {
          const int t = job_tile(jb, 0, s);
          if (!mbar_wait2_warp(&p_full[0], (sc0 + s) & 1u, &v_full[kv_stage(kt, t)], kv_phase(kt, t), abort_flag,
                               err, DEV_TIMEOUT_ATTN + 256 * 5, DEV_TIMEOUT_ATTN + 256 * 6)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(0, kv_stage(kt, t), s > 0, s + 1 == n0);
          if (!jb.pair) commit(&v_empty[kv_stage(kt, t)]);
          if (s + 1 < n0) {
            const int t2 = job_tile(jb, 0, s + 1);
            // no tcgen05 fence here: S reads only TMA-written Q and K (ordered
            // by their mbarrier), and it follows the PV block above, whose
            // fence already ordered the softmax's TMEM accesses, in issue order
            if (!wait_k(t2)) {
              ok = false;
              break;
            }
            issue_s(0, 0, kv_stage(kt, t2));
            if (!jb.pair) commit(&k_empty[kv_stage(kt, t2)]);
          }
        }
        if (s < n1) {
          // in a pair job, V tile t and K tile t2 are the ones warpgroup 0's
          // products above already waited for
          const int t = job_tile(jb, 1, s);
          if (!mbar_wait_warp(&p_full[1], (sc1 + s) & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 8) ||
              (!jb.pair && !wait_v(t))) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(1, kv_stage(kt, t), s > 0, s + 1 == n1);
          commit(&v_empty[kv_stage(kt, t)]);
          if (s + 1 < n1) {
            const int t2 = job_tile(jb, 1, s + 1);
            if (!jb.pair && !wait_k(t2)) {
              ok = false;
              break;
            }
            issue_s(1, qb1, kv_stage(kt, t2));
            commit(&k_empty[kv_stage(kt, t2)]);
          }
        }
      }
      // every MMA of this job issued: once they complete, Q may be reloaded
      commit(q_empty);
      sc0 += static_cast<uint32_t>(n0);
      sc1 += static_cast<uint32_t>(n1);
      kt += static_cast<uint32_t>(jb.nkv);
    }
    // every issued MMA has completed before TMEM is freed, also after an
    // abort (so this wait ignores the abort flag; it is bounded by time)
    commit(drain);
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(smem_u32(drain), 0u)) {
      if (globaltimer_ns() - t0 > HILO_WAIT_LIMIT_NS) {
        if (leader) atomicExch(err, DEV_TIMEOUT_ATTN + 256 * 9);
        break;
      }
    }
    __syncwarp();
    }
  } else {
    setmaxnreg_inc<SOFTMAX_REGS>();
    // ---------------- softmax: warpgroup i = warps 4i..4i+3, TMEM lane quarter warp % 4
    const int i = warp >> 2;
    const int row = (warp & 3) * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + 128u * i + lane_off;
    const uint32_t tO = tmem + 256u + 128u * i + lane_off;
    const uint32_t tO1 = tmem + 384u + lane_off;  // warpgroup 1's accumulator (split merge)
    // PROP: key weights of tile tt into the warp's slot `slot` (text tiles
    // weigh 1; columns past the ragged end 0), one commit group per call
    float* wslots = reinterpret_cast<float*>(smem + C::OFF_W) + warp * 2 * BKV;
    auto fetch_weights = [&](const Job& jb, int tt, int slot) {
      if (tt < jb.nkv) {
        float* wb = wslots + slot * BKV;
        if (tt < p.qt_txt) {
#pragma unroll
          for (int u = 0; u < 4; ++u) wb[lane + 32 * u] = 1.0f;
        } else {
          int r0, v;
          seq_tile(p, jb.b, jb.L, tt, r0, v);
          const float* src = p.n_img + (min(p.cu_img[jb.b], p.cap) + (tt - p.qt_txt) * BKV);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int col = lane + 32 * u;
            cp_async4(smem_u32(wb + col), col < v ? src + col : p.n_img, col < v ? 4u : 0u);
          }
        }
      }
      cp_async_commit();
    };
    bool ok = true;
    // sc*: S phases so far (one per step); oc*: o_done phases so far (one
    // per job in which the warpgroup has steps)
    uint32_t kt = 0, sc0 = 0, sc1 = 0, oc0 = 0, oc1 = 0;
    long long g = g_begin;
    Job jb;
    for (uint32_t jn = 0; ok && next_job(p, g, g_end, jb); ++jn) {
      const int n0 = job_steps(jb, 0), n1 = job_steps(jb, 1);
      const int n = i ? n1 : n0;
      const uint32_t sc = i ? sc1 : sc0;
      const uint32_t oc = i ? oc1 : oc0;
      float m = -INFINITY, l = 0.f;
      // ragged key tile: rows past `valid` hold other tokens (or stale data);
      // the warpgroup that owns V tile t (the first one in a pair) zeroes
      // them so that the zero-probability columns add exactly 0. Returns
      // false when the wait for V gave up.
      auto zero_v_tail = [&](int t, int valid) -> bool {
        if ((jb.pair ? i == 0 : true) && valid < BKV) {
          if (!mbar_wait_warp(&v_full[kv_stage(kt, t)], kv_phase(kt, t), abort_flag, err,
                              DEV_TIMEOUT_ATTN + 256 * 11))
            return false;
          if (row >= valid) {
            unsigned char* vr = sV(kv_stage(kt, t)) + row * 128;
#pragma unroll
            for (int j = 0; j < C::NBOX; ++j)
#pragma unroll
              for (int c16 = 0; c16 < 8; ++c16)
                *reinterpret_cast<uint4*>(vr + j * BOX_BYTES + c16 * 16) = make_uint4(0, 0, 0, 0);
          }
        }
        return true;
      };
      // S_i complete means every earlier MMA is too (PV_i of the previous
      // step included), so O_i can be rescaled and P_i written over S_i
      // without another wait. tcgen05.ld / tcgen05.st are warp-collective:
      // the whole warp rescales when any of its rows needs it (rows that do
      // not use alpha = 1)
      auto rescale_o = [&](bool rescale, float m_use) {
        if (__any_sync(0xffffffffu, rescale)) {
          const float alpha = rescale ? ex2(m - m_use) : 1.0f;
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            float o[32];
            tmem_ld32(tO + c * 32, o);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 32; ++j) o[j] *= alpha;
            tmem_st32(tO + c * 32, o);
          }
          l *= alpha;
        }
      };
      if (PROP && n > 0) fetch_weights(jb, job_tile(jb, i, 0), 0);
      for (int s = 0; s < n && ok; ++s) {
        const int t = job_tile(jb, i, s);
        int row0, valid;
        seq_tile(p, jb.b, jb.L, t, row0, valid);
        if (PROP) {
          // every lane is done with slot (s + 1) & 1 (read for step s - 1)
          // before the next step's weights are fetched into it
          __syncwarp();
          if (s + 1 < n) fetch_weights(jb, job_tile(jb, i, s + 1), (s + 1) & 1);
          else cp_async_commit();
        }
        if (!mbar_wait_warp(&s_full[i], (sc + s) & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 10)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // row max and row sum with 8 independent partials combined by a tree,
        // so the reductions do not form one 128-long dependent chain (the max
        // of a full tile takes two keys per three-input max); only the
        // last key tile of a segment is ragged and needs masking
        const bool full_tile = valid == BKV;
        float sv[BKV];
#pragma unroll
        for (int c = 0; c < BKV / 32; ++c) tmem_ld32(tS + c * 32, sv + c * 32);
        tmem_ld_wait();
        float mx8[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) mx8[u] = -INFINITY;
        if (full_tile) {
#pragma unroll
          for (int j = 0; j < BKV; j += 16)
#pragma unroll
            for (int u = 0; u < 8; ++u) mx8[u] = fmax3(mx8[u], sv[j + u], sv[j + 8 + u]);
        } else {
#pragma unroll
          for (int j = 0; j < BKV; ++j)
            if (j < valid) mx8[j & 7] = fmaxf(mx8[j & 7], sv[j]);
        }
        const float mx = fmax3(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(mx8[3], mx8[4], mx8[5]),
                               fmaxf(mx8[6], mx8[7]));
        const float m_tile = mx * p.scale_log2;
        bool rescale = false;
        float m_use = m;
        if (s == 0) {
          m_use = m_tile;
        } else if (m_tile > m + RESCALE_LOG2) {
          m_use = m_tile;
          rescale = true;
        }
        float ls8[8];
        if (PROP) {
          // probabilities by key pairs: exponent argument s*scale - m as one
          // paired fma, two exp2, times the pair's weights (one paired mul);
          // the row sum's partials (2u, 2u+1) for pair c with u = c mod 4 are
          // the same partition and order as key j into partial j mod 8.
          // Masked columns are 0, selected, never computed from their stale
          // logits. First: this step's weights have landed (all groups but
          // the newest) and are visible to the whole warp.
          cp_async_wait<1>();
          __syncwarp();
          const uint64_t* w2 = reinterpret_cast<const uint64_t*>(wslots + (s & 1) * BKV);
          const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-m_use, -m_use);
          uint64_t ls4[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) ls4[u] = 0ull;
#pragma unroll
          for (int c = 0; c < BKV / 2; ++c) {
            float a, a1;
            f2_split(f2_fma(f2(sv[2 * c], sv[2 * c + 1]), sc2, nm2), a, a1);
            a = (full_tile || 2 * c < valid) ? ex2(a) : 0.f;
            a1 = (full_tile || 2 * c + 1 < valid) ? ex2(a1) : 0.f;
            const uint64_t pr = f2_mul(f2(a, a1), w2[c]);
            f2_split(pr, sv[2 * c], sv[2 * c + 1]);
            ls4[c & 3] = f2_add(ls4[c & 3], pr);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) f2_split(ls4[u], ls8[2 * u], ls8[2 * u + 1]);
        } else {
#pragma unroll
          for (int u = 0; u < 8; ++u) ls8[u] = 0.f;
          if (full_tile) {
            // by key pairs: the exponent arguments as one paired fma, the
            // row-sum partials (2u, 2u+1) of pair c (u = c mod 4) as one
            // paired add; the same per-lane operations, partition and order
            // as key j into partial j mod 8 (one issue slot per pair)
            const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-m_use, -m_use);
            uint64_t ls4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) ls4[u] = 0ull;
#pragma unroll
            for (int c = 0; c < BKV / 2; ++c) {
              float a, a1;
              f2_split(f2_fma(f2(sv[2 * c], sv[2 * c + 1]), sc2, nm2), a, a1);
              a = ex2(a);
              a1 = ex2(a1);
              sv[2 * c] = a;
              sv[2 * c + 1] = a1;
              ls4[c & 3] = f2_add(ls4[c & 3], f2(a, a1));
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) f2_split(ls4[u], ls8[2 * u], ls8[2 * u + 1]);
          } else {
#pragma unroll
            for (int j = 0; j < BKV; ++j) {
              const float pj = j < valid ? ex2(fmaf(sv[j], p.scale_log2, -m_use)) : 0.f;
              sv[j] = pj;
              ls8[j & 7] += pj;
            }
          }
        }
        const float lsum =
            ((ls8[0] + ls8[1]) + (ls8[2] + ls8[3])) + ((ls8[4] + ls8[5]) + (ls8[6] + ls8[7]));
        if (!zero_v_tail(t, valid)) {
          ok = false;
          break;
        }
        rescale_o(rescale, m_use);
        m = m_use;
        l += lsum;
        // P_i as bf16 pairs (keys 2c, 2c+1 in column c) over the first 64
        // columns of S_i, the A operand of the PV product
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          float pk[32];
#pragma unroll
          for (int c = 0; c < 32; ++c)
            pk[c] = __uint_as_float(pack_bf16x2(sv[64 * h2 + 2 * c], sv[64 * h2 + 2 * c + 1]));
          tmem_st32(tS + 32 * h2, pk);
        }
        tmem_st_wait();
        // V rows zeroed above (ragged tile, owning warpgroup) are read by the
        // tensor core: make them visible to the async proxy before P_i is
        // handed over; other steps wrote no shared memory
        if ((jb.pair ? i == 0 : true) && valid < BKV) fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&p_full[i]);
      }
      if (PROP) cp_async_wait<0>();  // no copy in flight past this job
      // ---- output rows. A pair: warpgroup i writes query tile j0 + i. A
      // split job: warpgroup 1 hands its row maximum and sum to warpgroup 0,
      // which merges the two accumulators (each relative to its own maximum)
      // and writes query tile j0.
      const bool writer = jb.pair || i == 0;
      if (!jb.pair) {
        if (i == 1) {
          ml_slot[row] = m;
          ml_slot[BQ + row] = l;
        }
        named_bar_sync(1, 256);
      }
      float a0 = 1.f, a1 = 0.f, inv = 1.f;
      if (ok && writer) {
        bool done = mbar_wait_warp(&o_done[i], oc & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 14);
        if (!jb.pair && n1 > 0)
          done = done && mbar_wait_warp(&o_done[1], oc1 & 1u, abort_flag, err, DEV_TIMEOUT_ATTN + 256 * 15);
        ok = done;
        if (ok) {
          tc_fence_after();
          float lt = l;
          if (!jb.pair && n1 > 0) {
            const float m1 = ml_slot[row], l1 = ml_slot[BQ + row];
            const float mm = fmaxf(m, m1);
            a0 = ex2(m - mm);
            a1 = ex2(m1 - mm);
            lt = l * a0 + l1 * a1;
          }
          inv = 1.0f / lt;
          int qr0, qv;
          seq_tile(p, jb.b, jb.L, jb.j0 + (jb.pair ? i : 0), qr0, qv);
          // normalised O rows to bf16, staged through shared memory so that
          // the global stores leave as whole 128-byte lines (one row per
          // lane would write 16 bytes into 32 different rows per
          // instruction). Each warp owns a slice of the K stages: every S
          // product of the job, the last reader of K, completed before O did,
          // and the next job's K is loaded only after this job's epi_done.
          // The 16-byte units of a row are XOR-swizzled by the row, so neither
          // the writes (one row per lane) nor the reads (consecutive units of
          // a row) collide in the shared-memory banks.
          constexpr int UNITS = HD / 8;    // 16-byte units per row
          constexpr int RPI = 32 / UNITS;  // rows per store instruction
          uint4* stage = reinterpret_cast<uint4*>(smem + C::OFF_K) + warp * 32 * UNITS;
          const bool merge = !jb.pair && n1 > 0;
          auto stage_chunk = [&](int c, const float* o) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              uint4 v;
              v.x = pack_bf16x2(o[8 * j] * inv, o[8 * j + 1] * inv);
              v.y = pack_bf16x2(o[8 * j + 2] * inv, o[8 * j + 3] * inv);
              v.z = pack_bf16x2(o[8 * j + 4] * inv, o[8 * j + 5] * inv);
              v.w = pack_bf16x2(o[8 * j + 6] * inv, o[8 * j + 7] * inv);
              stage[lane * UNITS + ((4 * c + j) ^ (lane & (UNITS - 1)))] = v;
            }
          };
          if (!merge) {
            // all of O's columns in flight before one wait (the softmax's
            // registers are free here)
            float o[HD];
#pragma unroll
            for (int c = 0; c < HD / 32; ++c) tmem_ld32(tO + c * 32, o + c * 32);
#pragma unroll
            for (int c = 0; c < HD / 32; ++c) tmem_ld_wait_regs(o + c * 32);
#pragma unroll
            for (int c = 0; c < HD / 32; ++c) stage_chunk(c, o + c * 32);
          } else {
#pragma unroll 1
            for (int c = 0; c < HD / 32; ++c) {
              float o[32], o1[32];
              tmem_ld32(tO + c * 32, o);
              tmem_ld32(tO1 + c * 32, o1);
              tmem_ld_wait_regs(o);
              tmem_ld_wait_regs(o1);
#pragma unroll
              for (int j = 0; j < 32; ++j) o[j] = o[j] * a0 + o1[j] * a1;
              stage_chunk(c, o);
            }
          }
          __syncwarp();
          const int u = lane % UNITS;
#pragma unroll 4
          for (int k = 0; k < 32 / RPI; ++k) {
            const int rr = k * RPI + lane / UNITS;  // row within the warp's 32
            const int qrow = (warp & 3) * 32 + rr;  // row within the query tile
            if (qrow < qv)
              reinterpret_cast<uint4*>(p.out + static_cast<long long>(qr0 + qrow) * p.d + jb.h * HD)[u] =
                  stage[rr * UNITS + (u ^ (rr & (UNITS - 1)))];
          }
        }
      }
      // end of the job: the staging reads are done (generic proxy) before
      // the producer's next K copies (async proxy) overwrite the K stages;
      // in a split job warpgroup 1's accumulator has been read before its
      // next PV may overwrite it
      fence_proxy_async_smem();
      tc_fence_before();
      ok = bar_red_or(2, 256, !ok) ? false : ok;
      if (!ok) break;
      if (threadIdx.x == 0) mbar_arrive(epi_done);
      sc0 += static_cast<uint32_t>(n0);
      sc1 += static_cast<uint32_t>(n1);
      oc0 += n0 > 0 ? 1u : 0u;
      oc1 += n1 > 0 ? 1u : 0u;
      kt += static_cast<uint32_t>(jb.nkv);
    }
    if (PROP) cp_async_wait<0>();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, ATTN_TMEM_COLS);
  }
}

template <int HD, bool PROP>
cudaError_t launch_hd(const AttnArgs& a, const AttnParams& p, int grid, cudaStream_t st) {
  CUtensorMap tm;
  if (!encode_tmap_bf16_2d(&tm, a.qkv, 3ull * a.d, a.R, 3ull * a.d, 64, 128))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD, PROP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg<HD, PROP>::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  // the register split must fit what the CTA is launched with, or the
  // softmax warpgroups' setmaxnreg.inc would wait for registers forever
  static int regs = -1;
  if (regs < 0) {
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, attn_kernel<HD, PROP>);
    if (e != cudaSuccess) return e;
    regs = fa.numRegs;
  }
  if (static_cast<long long>(regs) * ATTN_THREADS < 256LL * SOFTMAX_REGS + 128LL * CONTROL_REGS)
    return cudaErrorInvalidConfiguration;
  return launch_pdl(attn_kernel<HD, PROP>, dim3(grid), dim3(ATTN_THREADS), Cfg<HD, PROP>::SMEM_BYTES, st, tm,
                    p);
}

}  // namespace

cudaError_t launch_attention(const AttnArgs& a, int num_sms, cudaStream_t st) {
  AttnParams p;
  p.cu_img = a.cu_img;
  p.n_img = a.n_img;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.B = a.B;
  p.T = a.T;
  p.heads = a.heads;
  p.d = a.d;
  p.qt_txt = (a.T + BQ - 1) / BQ;
  p.cap = a.R - a.B * a.T;
  p.scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(a.head_dim)));
  // a persistent grid: one CTA per SM; each takes its share of the query
  // tiles, whose count is known on the device only
  const int grid = num_sms > 0 ? num_sms : 1;
  if (a.n_img) {
    if (a.head_dim == 128) return launch_hd<128, true>(a, p, grid, st);
    if (a.head_dim == 64) return launch_hd<64, true>(a, p, grid, st);
    return cudaErrorInvalidValue;
  }
  if (a.head_dim == 128) return launch_hd<128, false>(a, p, grid, st);
  if (a.head_dim == 64) return launch_hd<64, false>(a, p, grid, st);
  return cudaErrorInvalidValue;
}

int attn_take_device_error() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(int)) != cudaSuccess) return -1;
  if (v) cudaMemcpyToSymbol(g_attn_err, &z, sizeof(int));
  return v;
}



}  // namespace hilo
