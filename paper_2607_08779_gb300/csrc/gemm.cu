// gemm.cu -- prefill GEMM over packed q-bit codes on the 5th-generation
// tensor cores (sm_103a: tcgen05 + tensor memory + TMA).
//
// Y[m][r] = sum_k w^[r][k] X[m][k]; in the prefill phase the matrix products
// set the time (Appendix B.2), and the
// symmetric formats compute only the integer-code GEMM term of the expansion
// in Appendix B.3 (the min-max grid adds the per-block minimum).
//
// Precision: the dequantised weight s*c is rounded to fp16 (<= 2^-11
// relative, where bf16 would give 2^-8 and miss the 1e-3 output gate) and
// the bf16 activations are converted to fp16 (exact for 2^-17 <= |x| <=
// 65504).  tcgen05.mma kind::f16 takes both operands in fp16 and accumulates
// in fp32 in tensor memory.
//
// Structure (one CTA per 128-row x BN-token output tile, 18 warps; the
// row tiles may belong to up to four matrices that share X, one launch for
// a fused q/k/v or gate/up projection):
//   warp 0     TMA producer for the fp16 activation tile (128B swizzle) and
//              owner of the tensor-memory allocation;
//   warp 1     a single elected thread issues tcgen05.mma (M=128, N=BN,
//              K=16 per instruction, 4 per 64-wide k-block) with the weight
//              operand A in tensor memory and the activations B in shared
//              memory, and commits to the stage's "empty" barrier;
//   warps 2-17 dequantise in two sets of eight that fill alternate stages:
//              each thread owns one weight row of the tile (its tensor-memory
//              lane) and one 32-code half of its set's 64-wide k-blocks,
//              loads those codes and their scale, forms fp16 s*c in natural
//              k order and writes it to the stage's A columns of tensor
//              memory with one tcgen05.st (shared memory then carries only
//              the activation tiles: the MMA's operand reads, the TMA writes
//              and no generic-proxy stores)
//              (a group whose scale lets s*c reach 65520, checked per scale
//              as |s| 2^(q-1) or |s| (2^q - 1) + |m|, raises SSS_FLAG_RANGE);
//              after the last k-block the same warps drain the fp32
//              accumulator with tcgen05.ld (each set of four warps one
//              quarter of the columns) and store Y (for a fixed token, a warp writes
//              32 consecutive floats).
// Tensor memory (512 columns): the fp32 accumulator in columns [0, BN), the
// A stages in columns BN + 32 s (one 64-wide fp16 k-block of 128 rows per
// 32 columns: lane = row, two k-consecutive halves per 32-bit column).
// Every mbarrier wait is bounded (about one second of global time); on
// expiry the CTA raises SSS_FLAG_TIMEOUT, all roles leave their loops, and
// the tensor memory is still released.
#include <cuda.h>

#include <string.h>

#include <algorithm>
#include <mutex>

#include "sss_internal.cuh"

namespace sss {
namespace {

constexpr int kBM = 128;            // weight rows per tile (MMA M)
constexpr int kBK = 64;             // k per stage (128 bytes of fp16)
constexpr int kDqWarps = 8;         // warps that fill one stage
// threads of a CTA with SETS sets of 8 dequantising warps (on alternate
// k-blocks), the producer warp and the MMA issuer's warp
template <int SETS>
constexpr int threads_of() { return 64 + 32 * kDqWarps * SETS; }
constexpr uint64_t kWaitNs = 1000000000ull;  // bounded waits: 1 s

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on a phase parity.  Returns false when the wait gave up,
// either on its own time limit or because another role raised *abort.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity,
                                          volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort) return false;
      if (global_ns() - t0 > kWaitNs) {
        *abort = 1;
        return false;
      }
    }
  }
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(const CUtensorMap* map, uint64_t* bar, void* dst,
                                            int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}

// tcgen05 shared-memory matrix descriptor: K-major operand, 128-byte swizzle,
// 8-row swizzle atoms 1024 bytes apart (stride byte offset), descriptor
// version 1 at bit 46.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);          // start address
  d |= static_cast<uint64_t>(1) << 16;                           // LBO (unused for SW128 K-major)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;                    // SBO: 1024 B
  d |= static_cast<uint64_t>(1) << 46;                           // version
  d |= static_cast<uint64_t>(2) << 61;                           // 128B swizzle
  return d;
}

// Instruction descriptor, kind::f16: D fp32, A and B fp16, both K-major.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N) {
  return (1u << 4)                                    // D format: F32
         | (0u << 7) | (0u << 10)                     // A, B format: F16
         | (static_cast<uint32_t>(N >> 3) << 17)      // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);     // M / 16
}

// The four MMAs of one 64-wide k-block (K = 16 each) in one block: A from
// tensor memory at a_tmem + 8 kk, B from the swizzled shared tile whose
// descriptor is b_desc + 2 kk (32 bytes further along k; the start-address
// field counts 16-byte units and does not carry), accumulating into d_tmem
// unless first is set (the tile's first k-block starts from zero).
__device__ __forceinline__ void umma_kblock(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t first) {
  asm volatile(
      "{\n .reg .pred p;\n setp.eq.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%5], %6, %3, 1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%7], %8, %3, 1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%9], %10, %3, 1;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(first), "r"(a_tmem + 8), "l"(b_desc + 2),
      "r"(a_tmem + 16), "l"(b_desc + 4), "r"(a_tmem + 24), "l"(b_desc + 6)
      : "memory");
}
// 16 consecutive 32-bit columns of the warp's 32 lanes
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Dequantisation of 32 codes of one row into 16 natural-order fp16 pairs.
// ---------------------------------------------------------------------------

// PRMT selector: result = [a.byte_i, 0, b.byte_i, 0]; the zero bytes use the
// sign-replicate mode on a byte whose top bit is clear.
__device__ __forceinline__ uint32_t pair_bytes(uint32_t a, uint32_t b, int i) {
  const uint32_t sel = static_cast<uint32_t>(i) | (static_cast<uint32_t>(8 + i) << 4) |
                       (static_cast<uint32_t>(4 + i) << 8) |
                       (static_cast<uint32_t>(12 + i) << 12);
  uint32_t r;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
  return r;
}

// u pairs (natural order: element 2p in the low half, 2p+1 in the high half)
// of a 32-code sub-chunk, as 16-bit integers.
template <int Q>
__device__ __forceinline__ void code_pairs(const uint32_t* w, uint32_t (&u)[16]) {
  if constexpr (Q == 4) {
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
      const uint32_t ev = w[wi] & 0x0F0F0F0Fu, od = (w[wi] >> 4) & 0x0F0F0F0Fu;
#pragma unroll
      for (int i = 0; i < 4; ++i) u[4 * wi + i] = pair_bytes(ev, od, i);
    }
  } else {
#pragma unroll
    for (int wi = 0; wi < 2; ++wi) {
      const uint32_t a = w[wi] & 0x03030303u, b = (w[wi] >> 2) & 0x03030303u;
      const uint32_t c = (w[wi] >> 4) & 0x03030303u, d = (w[wi] >> 6) & 0x03030303u;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        u[8 * wi + 2 * i] = pair_bytes(a, b, i);
        u[8 * wi + 2 * i + 1] = pair_bytes(c, d, i);
      }
    }
    if constexpr (Q == 3) {
      const uint32_t hi = w[2];
#pragma unroll
      for (int p = 0; p < 16; ++p) {
        const uint32_t v = (hi >> (2 * p)) & 3u;
        u[p] |= ((v & 1u) << 2) | ((v & 2u) << 17);  // + 4*hi bit, both halves
      }
    }
  }
}

template <int Q>
__device__ __forceinline__ void load_sub32(const uint8_t* __restrict__ row, int64_t grp, int sc,
                                           int G, bool valid, uint32_t* w) {
  if constexpr (Q == 4) {
    uint4 v = make_uint4(0, 0, 0, 0);
    if (valid) v = __ldcs(reinterpret_cast<const uint4*>(row + grp * (G / 2) + sc * 16));
    w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
  } else if constexpr (Q == 2) {
    uint2 v = make_uint2(0, 0);
    if (valid) v = __ldcs(reinterpret_cast<const uint2*>(row + grp * (G / 4) + sc * 8));
    w[0] = v.x; w[1] = v.y;
  } else {
    w[0] = w[1] = w[2] = 0;
    if (valid) {
      const uint32_t* base = reinterpret_cast<const uint32_t*>(row + grp * (3 * G / 8));
      w[0] = __ldcs(base + 2 * sc);
      w[1] = __ldcs(base + 2 * sc + 1);
      w[2] = __ldcs(base + G / 16 + sc);
    }
  }
}

// One weight matrix of a call (several share X, e.g. a fused q/k/v
// projection): its row tiles are tiles tile0 .. tile0 + ceil(n / 128) - 1 of
// the grid's x dimension.
struct GemmJob {
  const uint8_t* codes;
  const uint16_t* scales;
  const uint16_t* mins;
  float* y;  // [m][n]
  int64_t n;
  int64_t tile0;
};
struct GemmArgs {
  GemmJob job[kMaxGemmJobs];
  int njobs;
  uint32_t* status;
  int64_t m, k;
  int G;
  int stall;  // test hook: the first stage's weight tile is never announced
  // split K: CTA z of nsplit takes k-blocks [z * chunk, ...) and leaves its
  // fp32 tile in part + z * m * np (row tile t at rows 128 t .. 128 t + 127
  // of np = 128 x all row tiles); the last of a tile's splits to finish
  // (counted in cnt, zero on entry) sums them in split order into y
  int nsplit;
  int64_t np;
  float* part;
  int* cnt;
};

// The activation tile map, and per matrix its code and scale tile maps
// (used with TW).
struct GemmMaps {
  CUtensorMap x;
  CUtensorMap c[kMaxGemmJobs];
  CUtensorMap s[kMaxGemmJobs];
};

// Shared memory: STAGES activation tiles (1024-aligned for the 128-byte
// swizzle), then with TW the stages' packed-code tiles (128 rows x 8q bytes)
// and scale windows (128 rows x 8 fp16), then the barriers.
template <int BN, int STAGES, int Q, bool TW>
struct Smem {
  static constexpr int B_BYTES = BN * kBK * 2;               // 16 or 32 KB
  static constexpr int C_BYTES = TW ? kBM * 8 * Q : 0;       // codes of one k-block
  static constexpr int S_BYTES = TW ? kBM * 16 : 0;          // 8 scales per row
  static constexpr int STAGE = B_BYTES;
  static constexpr int C_OFF = STAGES * B_BYTES;
  static constexpr int S_OFF = C_OFF + STAGES * C_BYTES;
  static constexpr int BAR_OFF = S_OFF + STAGES * S_BYTES;
  static constexpr int TOTAL = BAR_OFF + (3 * STAGES + 1) * 8 + 16 + 1024;  // + align slack
  static constexpr int A_COL = BN;                // first A-stage column in tensor memory
  static_assert(TOTAL <= 227 * 1024, "shared memory per CTA");
};
// tensor-memory columns a CTA allocates: all 512 with one CTA per SM, half
// when two CTAs (one dequantising set each) share an SM
template <int SETS>
constexpr int tmem_cols_of() { return SETS == 1 ? 256 : 512; }

// TW: the packed codes and scales arrive by TMA with the activation tile
// (q = 2, 4 on the symmetric grids, where a k-block's codes are 16-byte
// aligned); otherwise each dequantising thread loads its own from global
// memory a few k-blocks ahead.
template <int Q, bool ASYM, int BN, int STAGES, bool TW, int SETS>
__global__ void __launch_bounds__(threads_of<SETS>(), SETS == 1 ? 2 : 1)
    gemm_kernel(const __grid_constant__ GemmMaps maps, const __grid_constant__ GemmArgs a) {
  using S = Smem<BN, STAGES, Q, TW>;
  constexpr int kTmemCols = tmem_cols_of<SETS>();
  static_assert(BN + 32 * STAGES <= kTmemCols, "tensor memory holds the accumulator and A stages");
  extern __shared__ unsigned char smem_raw[];
  // 1024-byte alignment for the swizzle atoms
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full_a = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF);
  uint64_t* full_b = full_a + STAGES;
  uint64_t* empty = full_b + STAGES;
  uint64_t* done = empty + STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // this CTA's matrix jb, its rows n0 .. n0 + 127 in that matrix, and the
  // same rows g0 .. g0 + 127 of the partial tiles
  int jb = 0;
  while (jb + 1 < a.njobs && static_cast<int64_t>(blockIdx.x) >= a.job[jb + 1].tile0) ++jb;
  const GemmJob& job = a.job[jb];
  const int64_t n0 = (static_cast<int64_t>(blockIdx.x) - job.tile0) * kBM;
  const int64_t g0 = static_cast<int64_t>(blockIdx.x) * kBM;
  const int64_t m0 = static_cast<int64_t>(blockIdx.y) * BN;
  // this split's k-blocks: global k-block kb_base + kb for kb = 0 .. nkb - 1
  const int nkb_all = static_cast<int>(a.k / kBK);
  const int chunk = (nkb_all + a.nsplit - 1) / a.nsplit;
  const int kb_base = static_cast<int>(blockIdx.z) * chunk;
  const int nkb = min(nkb_all - kb_base, chunk);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_a[s], kDqWarps);
      mbar_init(&full_b[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    *abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Launched as a programmatic dependent launch: the set-up above (barriers,
  // tensor memory) overlaps the preceding kernel's drain; nothing in global
  // memory is read or written before that kernel has completed.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");

  if (warp == 0) {
    // ---------------- TMA producer: activation tiles ----------------
    if (lane == 0) {
      int issued = 0;
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = static_cast<uint32_t>(kb / STAGES) & 1u;
        if (!mbar_wait(&empty[s], ph ^ 1u, abort)) break;
        unsigned char* sb = smem + s * S::STAGE;
        mbar_arrive_expect_tx(&full_b[s], S::B_BYTES + S::C_BYTES + S::S_BYTES);
        tma_load_2d(&maps.x, &full_b[s], sb, (kb_base + kb) * kBK, static_cast<int>(m0));
        if constexpr (TW) {
          // the k-block's codes (8q bytes of each row, x a multiple of 16) and
          // the 8-scale window holding its groups (x rounded down to 8)
          tma_load_2d(&maps.c[jb], &full_b[s], smem + S::C_OFF + s * S::C_BYTES,
                      (kb_base + kb) * 8 * Q, static_cast<int>(n0));
          tma_load_2d(&maps.s[jb], &full_b[s], smem + S::S_OFF + s * S::S_BYTES,
                      ((kb_base + kb) * kBK / a.G) & ~7, static_cast<int>(n0));
        }
        issued = kb + 1;
      }
      if (*abort) {
        // let this CTA's copies still in flight land before the CTA exits
        int drain = 0;
        for (int kb = std::max(0, issued - STAGES); kb < issued; ++kb)
          (void)mbar_wait(&full_b[kb % STAGES], static_cast<uint32_t>(kb / STAGES) & 1u, &drain);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc = make_idesc(kBM, BN);
      // stage s: A at tensor-memory column A_COL + 32 s, B at shared offset
      // s * STAGE (its descriptor's start-address field moves by STAGE / 16)
      const uint32_t ta0 = tmem + static_cast<uint32_t>(S::A_COL);
      const uint64_t bdesc0 = sw128_desc(smem_u32(smem));
      constexpr uint64_t bstep = static_cast<uint64_t>(S::STAGE >> 4);
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = static_cast<uint32_t>(kb / STAGES) & 1u;
        if (!mbar_wait(&full_a[s], ph, abort)) break;
        if (!mbar_wait(&full_b[s], ph, abort)) break;
        tc_fence_after();
        umma_kblock(tmem, ta0 + static_cast<uint32_t>(32 * s), bdesc0 + bstep * s, idesc,
                    kb == 0 ? 1u : 0u);
        umma_commit(&empty[s]);  // frees the stage once these MMAs complete
      }
      umma_commit(done);
    }
  } else {
    // ---------------- dequantise, then epilogue ----------------
    // a warp may touch tensor-memory lanes 32*(warp % 4) .. +31 only, so
    // thread (warp, lane) owns tile row 32*(warp % 4) + lane; the dequant
    // warps w = warp - 2 form four groups of four (w >> 2), each covering
    // the 128 rows once: group g takes the 32-code half hf = g & 1 of the
    // k-blocks kb = set, set + SETS, ... of set g >> 1
    const int row_i = 32 * (warp & 3) + lane;
    const int hf = ((warp - 2) >> 2) & 1;
    const int set = (warp - 2) >> 3;
    bool big = false;  // a group whose s*c may leave the fp16 range
    bool ok = true;
    // fp16 s*c (ASYM: s*u + m) of the thread's 32 codes w into stage s's A
    // columns 16 hf .. 16 hf + 15 of lane row_i, then the arrive
    auto emit = [&](const uint32_t* w, uint16_t s16, uint16_t m16, int s, int kb) {
      {
        const __half sh = __ushort_as_half(s16);
        const __half2 s2 = __halves2half2(sh, sh);
        __half2 m2 = __float2half2_rn(0.f);
        const float sa = fabsf(__half2float(sh));
        if constexpr (!ASYM) big |= sa * static_cast<float>(1 << (Q - 1)) >= 65520.f;
        if constexpr (ASYM) {
          const __half mh = __ushort_as_half(m16);
          m2 = __halves2half2(mh, mh);
          big |= sa * static_cast<float>((1 << Q) - 1) + fabsf(__half2float(mh)) >= 65520.f;
        }
        uint32_t u[16];
        code_pairs<Q>(w, u);
        uint32_t out[16];
#pragma unroll
        for (int p = 0; p < 16; ++p) {
          // 1024 + u as fp16, minus 1024 (+ 2^(q-1) for symmetric codes): exact
          const uint32_t mag = u[p] | 0x64006400u;
          __half2 hv = *reinterpret_cast<const __half2*>(&mag);
          const __half2 bias = ASYM ? __float2half2_rn(1024.f)
                                    : __float2half2_rn(static_cast<float>(1024 + (1 << (Q - 1))));
          hv = __hsub2(hv, bias);                               // c (or u) exactly
          hv = ASYM ? __hfma2(hv, s2, m2) : __hmul2(hv, s2);    // RN16(s*c) / RN16(s*u+m)
          out[p] = *reinterpret_cast<const uint32_t*>(&hv);
        }
        tmem_st16(tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16) +
                      static_cast<uint32_t>(S::A_COL + 32 * s + 16 * hf),
                  out);
      }
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      tc_fence_before();  // the stores, then the arrive the MMA issuer waits on
      __syncwarp();
      // (sss_test_set_stall: warp 2 leaves the first stage one arrive
      // short, so the MMA issuer's wait for it runs out)
      if (lane == 0 && !(a.stall && kb == 0 && warp == 2)) mbar_arrive(&full_a[s]);
    };
    if constexpr (TW) {
      for (int kb = set; kb < nkb; kb += SETS) {
        const int s = kb % STAGES;
        const uint32_t ph = static_cast<uint32_t>(kb / STAGES) & 1u;
        // warp-uniform, since the tensor-memory stores are .sync.aligned:
        // the stage's A columns are free and its code and scale tiles landed
        const bool freed = mbar_wait(&empty[s], ph ^ 1u, abort);
        if (!__all_sync(0xffffffffu, freed)) {
          ok = false;
          break;
        }
        const bool landed = mbar_wait(&full_b[s], ph, abort);
        if (!__all_sync(0xffffffffu, landed)) {
          ok = false;
          break;
        }
        tc_fence_after();  // the MMAs that read this stage have completed
        const unsigned char* cs = smem + S::C_OFF + s * S::C_BYTES + row_i * (8 * Q) + hf * (4 * Q);
        uint32_t w[4] = {0u, 0u, 0u, 0u};
        if constexpr (Q == 4) {
          const uint4 v = *reinterpret_cast<const uint4*>(cs);
          w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
        } else {
          const uint2 v = *reinterpret_cast<const uint2*>(cs);
          w[0] = v.x; w[1] = v.y;
        }
        const int kg = kb_base + kb;
        const int gi = (kg * kBK + 32 * hf) / a.G, g0 = (kg * kBK / a.G) & ~7;
        const uint16_t s16 = *reinterpret_cast<const uint16_t*>(
            smem + S::S_OFF + s * S::S_BYTES + row_i * 16 + 2 * (gi - g0));
        emit(w, s16, 0, s, kb);
      }
    } else {
      const int64_t r = n0 + row_i;
      const bool rok = r < job.n;
      const int64_t nG = a.k / a.G;
      const uint8_t* rowp = job.codes + (rok ? r : 0) * (a.k * Q / 8);
      // codes and scale (and min) of this thread's half of one k-block
      struct KBlock {
        uint32_t w[4];
        uint16_t s, m;
      };
      auto fetch = [&](KBlock& d, int kb) {
        if (kb >= nkb) return;
        const int64_t kc = static_cast<int64_t>(kb_base + kb) * kBK + 32 * hf;
        const int64_t grp = kc / a.G;
        const int sc = static_cast<int>((kc % a.G) / 32);
        load_sub32<Q>(rowp, grp, sc, a.G, rok, d.w);
        d.s = rok ? __ldcs(job.scales + r * nG + grp) : static_cast<uint16_t>(0);
        if constexpr (ASYM) d.m = rok ? __ldcs(job.mins + r * nG + grp) : static_cast<uint16_t>(0);
      };
      // the global loads run kPrefetch of this thread's k-blocks ahead of use
      constexpr int kPrefetch = 4;
      KBlock ring[kPrefetch];
#pragma unroll
      for (int q0 = 0; q0 < kPrefetch; ++q0) fetch(ring[q0], set + SETS * q0);
      for (int kb0 = set; kb0 < nkb && ok; kb0 += SETS * kPrefetch) {
#pragma unroll
        for (int q0 = 0; q0 < kPrefetch; ++q0) {
          const int kb = kb0 + SETS * q0;
          if (kb >= nkb || !ok) break;
          const int s = kb % STAGES;
          const uint32_t ph = static_cast<uint32_t>(kb / STAGES) & 1u;
          // warp-uniform, since the tensor-memory stores are .sync.aligned
          const bool freed = mbar_wait(&empty[s], ph ^ 1u, abort);
          if (!__all_sync(0xffffffffu, freed)) {
            ok = false;
            break;
          }
          tc_fence_after();  // the MMAs that read this stage have completed
          emit(ring[q0].w, ring[q0].s, ring[q0].m, s, kb);
          fetch(ring[q0], kb + SETS * kPrefetch);
        }
      }
    }
    if (__any_sync(0xffffffffu, big) && lane == 0 && a.status != nullptr)
      atomicOr(a.status, SSS_FLAG_RANGE);
    // ---------------- epilogue ----------------
    // a warp may read tensor-memory lanes 32*(warp % 4) .. +31; the four
    // sets of four warps take one quarter of the columns each
    const bool fin = ok && mbar_wait(done, 0, abort);
    if (__all_sync(0xffffffffu, fin)) {  // warp-uniform: tcgen05.ld is .sync.aligned
      tc_fence_after();
      const int sub = warp & 3;
      const int row_local = sub * 32 + lane;
      const int64_t rr = n0 + row_local;
      constexpr int kCols = BN / (kDqWarps * SETS / 4);
      const int cbeg = ((warp - 2) >> 2) * kCols;
#pragma unroll 1
      for (int c0 = cbeg; c0 < cbeg + kCols; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(tmem + (static_cast<uint32_t>(sub * 32) << 16) + c0, v);
        // one split: y; several: this split's partial tile
        const bool split = a.nsplit > 1;
        float* dst = split ? a.part + static_cast<int64_t>(blockIdx.z) * a.m * a.np + g0 + row_local
                           : job.y + rr;
        const int64_t ld = split ? a.np : job.n;
        if (rr < job.n) {
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const int64_t mm = m0 + c0 + c;
            if (mm < a.m) dst[mm * ld] = __uint_as_float(v[c]);
          }
        }
      }
    }
  }

  if (a.nsplit > 1) __threadfence();  // this CTA's partial tile, device-wide
  tc_fence_before();
  __syncthreads();
  if (*abort && threadIdx.x == 0 && a.status != nullptr) atomicOr(a.status, SSS_FLAG_TIMEOUT);
  if (a.nsplit > 1 && !*abort) {
    // the tile's last split to arrive sums the partials in split order
    // (z = 0, 1, ...: the same order whichever split is last) into y and
    // leaves the counter at zero
    int* cnt = a.cnt + blockIdx.y * gridDim.x + blockIdx.x;
    volatile int* last = abort + 1;
    if (threadIdx.x == 0) *last = atomicAdd(cnt, 1) == a.nsplit - 1;
    __syncthreads();
    if (*last) {
      __threadfence();
      // 4 consecutive rows per element (n % 4 == 0, y and the partials
      // 16-byte aligned); eight elements per thread at a time, so every
      // split's eight loads are in flight together
      constexpr int kV = kBM / 4;  // float4 per token of the tile
      constexpr int kE = 8;
      const int64_t mn = a.m * a.np;
      for (int e0 = threadIdx.x; e0 < kV * BN; e0 += kE * blockDim.x) {
        float4 acc[kE];
        int64_t off[kE];
        bool in[kE];
#pragma unroll
        for (int j = 0; j < kE; ++j) {
          const int e = e0 + j * blockDim.x;
          const int64_t mm = m0 + e / kV, rr = n0 + 4 * (e % kV);
          in[j] = e < kV * BN && mm < a.m && rr < job.n;
          off[j] = in[j] ? mm * a.np + g0 + 4 * (e % kV) : 0;
          acc[j] = in[j] ? __ldcg(reinterpret_cast<const float4*>(a.part + off[j]))
                         : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        for (int z = 1; z < a.nsplit; ++z) {
          float4 v[kE];
#pragma unroll
          for (int j = 0; j < kE; ++j)
            v[j] = in[j] ? __ldcg(reinterpret_cast<const float4*>(a.part + z * mn + off[j]))
                         : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int j = 0; j < kE; ++j) {
            acc[j].x += v[j].x; acc[j].y += v[j].y; acc[j].z += v[j].z; acc[j].w += v[j].w;
          }
        }
#pragma unroll
        for (int j = 0; j < kE; ++j) {
          const int e = e0 + j * blockDim.x;
          if (in[j])
            *reinterpret_cast<float4*>(job.y + (m0 + e / kV) * job.n + n0 + 4 * (e % kV)) = acc[j];
        }
      }
      if (threadIdx.x == 0) *cnt = 0;
    }
  }
  if (warp == 0) {
    tc_fence_after();
    if (*abort) {  // MMAs still in flight must retire before the TMEM is released
      int drain = 0;
      (void)mbar_wait(done, 0, &drain);
    }
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

// bf16 -> fp16 activation conversion (round to nearest even)
__global__ void __launch_bounds__(256)
    bf16_to_f16_kernel(const uint16_t* __restrict__ x, __half* __restrict__ y, int64_t nvec) {
  // programmatic dependent launch: start once the preceding kernel (which
  // may still read the fp16 buffer) has completed
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += stride) {
    const uint4 v = __ldcs(reinterpret_cast<const uint4*>(x) + i);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float lo = __uint_as_float(w[e] << 16);
      const float hi = __uint_as_float(w[e] & 0xFFFF0000u);
      __half2 h = __floats2half2_rn(lo, hi);
      o[e] = *reinterpret_cast<uint32_t*>(&h);
    }
    reinterpret_cast<uint4*>(y)[i] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

// bytes of the fp16 copy of X, rounded up to 256; SIZE_MAX when m * k * 2
// does not fit in size_t (such a call is rejected before it gets here)
size_t x16_bytes(int64_t m, int64_t k) {
  if (m < 0 || k < 0) return SIZE_MAX;
  const size_t mm = static_cast<size_t>(m), kk = static_cast<size_t>(k);
  if (kk != 0 && mm > (SIZE_MAX - 255) / 2 / kk) return SIZE_MAX;
  return (mm * kk * 2 + 255) / 256 * 256;
}

// How a call runs: tile width, dequantising sets per CTA, K splits.
struct GemmPlan {
  int bn, sets, nsplit;
};

// Workspace layout: fp16 X, then (split K) the partial tiles (rows padded to
// whole row tiles, rt of them over all the call's matrices), then the
// per-tile counters.
size_t round256(size_t b) { return (b + 255) / 256 * 256; }
size_t split_bytes(int64_t rt, int64_t m, const GemmPlan& p) {
  if (p.nsplit <= 1) return 0;
  const size_t tiles = static_cast<size_t>(rt) * ((m + p.bn - 1) / p.bn);
  return round256(static_cast<size_t>(p.nsplit) * m * rt * kBM * 4) + round256(tiles * 4);
}

// Largest K split (>= 2 to count) that fills the idle SMs with `tiles`
// tiles, keeps every split non-empty and at least `min_kb` k-blocks long,
// and whose partial tiles fit in the workspace (ws bytes); 1 if none.
int split_for(int64_t k, int64_t rt, int64_t m, size_t ws, int bn, int64_t tiles, int64_t min_kb) {
  const int64_t sms = device_sm_count();
  const int64_t nkb = k / kBK;
  int split = static_cast<int>(std::min<int64_t>(sms / std::max<int64_t>(tiles, 1), nkb / min_kb));
  if (split >= 2) {  // every split non-empty: as many as chunks of ceil(nkb / split)
    const int64_t chunk = (nkb + split - 1) / split;
    split = static_cast<int>((nkb + chunk - 1) / chunk);
  }
  for (; split >= 2; --split) {
    const GemmPlan p{bn, 2, split};
    if (x16_bytes(m, k) <= ws && x16_bytes(m, k) + split_bytes(rt, m, p) <= ws) return split;
  }
  return 1;
}

// 256-token tiles when they cover the SMs (each weight tile is then
// dequantised for twice the tokens, and a k-block's MMAs take about as long
// at N = 256 as at N = 128).  Otherwise, when each split keeps at least 64
// k-blocks, 256-token tiles with K split over as many CTAs as fill the SMs;
// else 256-token tiles unsplit when 128-token tiles would need a second
// wave; else 128-token tiles, split (at least 8 k-blocks each) when they
// leave SMs idle.  The tile's last split sums all partials alone, so a split pays
// only with enough k-blocks behind it.  (Two half-size CTAs per SM, one
// dequantising set each, measured slower than one full CTA: their rings are
// half as deep.)  rt: the row tiles of all the call's matrices.
GemmPlan plan_gemm(int64_t rt, int64_t k, int64_t m, size_t ws) {
  const int64_t sms = device_sm_count();
  if (m > 128) {
    const int64_t tiles = rt * ((m + 255) / 256);
    if (tiles >= sms) return {256, 2, 1};
    const int split = split_for(k, rt, m, ws, 256, tiles, 64);
    if (split >= 2) return {256, 2, split};
    // 128-token tiles would take a second wave (each CTA the whole k-range
    // again) where 256-token tiles take one
    if (rt * ((m + 127) / 128) > sms) return {256, 2, 1};
  }
  const int64_t tiles = rt * ((m + 127) / 128);
  if (tiles >= sms) return {128, 2, 1};
  return {128, 2, split_for(k, rt, m, ws, 128, tiles, 8)};
}

int64_t row_tiles(const sss_qtensor_t* const* ts, int count) {
  int64_t rt = 0;
  for (int j = 0; j < count; ++j) rt += (ts[j]->n + kBM - 1) / kBM;
  return rt;
}

template <int Q, bool ASYM, int BN, bool TW, int SETS>
cudaError_t run_gemm(const sss_qtensor_t* const* ts, float* const* ys, int count,
                     const __half* x16, int64_t m, uint32_t* status, cudaStream_t stream,
                     int nsplit, unsigned char* ws_split) {
  constexpr int STAGES = (BN == 256) ? (TW ? 5 : 6) : 8;
  using S = Smem<BN, STAGES, Q, TW>;
  const sss_qtensor_t& t0 = *ts[0];  // k, q, group and grid are those of every matrix
  EncodeTiledFn enc = tensor_map_encoder();
  if (enc == nullptr) return cudaErrorNotSupported;
  GemmMaps maps;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(t0.k), static_cast<cuuint64_t>(m)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(t0.k) * 2};
  const cuuint32_t box[2] = {kBK, BN};
  const cuuint32_t estr[2] = {1, 1};
  CUresult cr = enc(&maps.x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half*>(x16), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;
  GemmArgs a;
  memset(&a, 0, sizeof a);
  int64_t tile0 = 0;
  for (int j = 0; j < count; ++j) {
    const sss_qtensor_t& t = *ts[j];
    maps.c[j] = maps.x;  // placeholders unless TW
    maps.s[j] = maps.x;
    if constexpr (TW) {
      // packed codes [n][k q / 8] bytes: one k-block is 8q bytes of 128 rows;
      // scales [n][k / G] fp16: a window of 8 (16 bytes) of 128 rows; rows
      // past n read as zero
      const cuuint64_t cd[2] = {static_cast<cuuint64_t>(t.k * Q / 8), static_cast<cuuint64_t>(t.n)};
      const cuuint64_t cs[1] = {static_cast<cuuint64_t>(t.k * Q / 8)};
      const cuuint32_t cb[2] = {static_cast<cuuint32_t>(8 * Q), kBM};
      cr = enc(&maps.c[j], CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, t.codes, cd, cs, cb, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;
      const int64_t ng = t.k / t.group;
      const cuuint64_t sd[2] = {static_cast<cuuint64_t>(ng), static_cast<cuuint64_t>(t.n)};
      const cuuint64_t ss[1] = {static_cast<cuuint64_t>(ng * 2)};
      const cuuint32_t sbx[2] = {8, kBM};
      cr = enc(&maps.s[j], CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, t.scales, sd, ss, sbx, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    a.job[j].codes = t.codes;
    a.job[j].scales = t.scales;
    a.job[j].mins = t.mins;
    a.job[j].y = ys[j];
    a.job[j].n = t.n;
    a.job[j].tile0 = tile0;
    tile0 += (t.n + kBM - 1) / kBM;
  }
  auto kern = gemm_kernel<Q, ASYM, BN, STAGES, TW, SETS>;
  cudaError_t e = ensure_smem(kern, S::TOTAL);
  if (e != cudaSuccess) return e;
  a.njobs = count;
  a.status = status;
  a.m = m;
  a.k = t0.k;
  a.G = t0.group;
  a.stall = (test_stall_mask() & SSS_TEST_STALL_GEMM) ? 1 : 0;
  a.nsplit = nsplit;
  a.np = tile0 * kBM;
  a.part = nullptr;
  a.cnt = nullptr;
  const unsigned gx = static_cast<unsigned>(tile0);
  const unsigned gy = static_cast<unsigned>((m + BN - 1) / BN);
  if (nsplit > 1) {
    a.part = reinterpret_cast<float*>(ws_split);
    a.cnt = reinterpret_cast<int*>(ws_split + round256(static_cast<size_t>(nsplit) * m * a.np * 4));
    e = cudaMemsetAsync(a.cnt, 0, sizeof(int) * gx * gy, stream);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(gx, gy, static_cast<unsigned>(nsplit));
  cfg.blockDim = dim3(threads_of<SETS>(), 1, 1);
  cfg.dynamicSmemBytes = S::TOTAL;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, maps, a);
}

struct GemmCall {
  const sss_qtensor_t* const* ts;
  float* const* ys;
  int count;
  const __half* x16;
  int64_t m;
  uint32_t* status;
  cudaStream_t stream;
  GemmPlan plan;
  unsigned char* ws_split;
};

template <int Q, bool ASYM, bool TW>
cudaError_t gemm_tw(const GemmCall& c) {
  if (c.plan.bn == 256)
    return run_gemm<Q, ASYM, 256, TW, 2>(c.ts, c.ys, c.count, c.x16, c.m, c.status, c.stream,
                                         c.plan.nsplit, c.ws_split);
  return run_gemm<Q, ASYM, 128, TW, 2>(c.ts, c.ys, c.count, c.x16, c.m, c.status, c.stream,
                                       c.plan.nsplit, c.ws_split);
}

template <int Q, bool ASYM>
cudaError_t gemm_bn(const GemmCall& c) {
  if constexpr (!ASYM && Q != 3) {
    // the code and scale tiles by TMA: 16-byte aligned scale rows in every
    // matrix
    bool tw = ((c.ts[0]->k / c.ts[0]->group) * 2) % 16 == 0;
    for (int j = 0; j < c.count; ++j)
      tw = tw && (reinterpret_cast<uintptr_t>(c.ts[j]->scales) % 16) == 0;
    if (tw) return gemm_tw<Q, ASYM, true>(c);
  }
  return gemm_tw<Q, ASYM, false>(c);
}

template <int Q>
cudaError_t gemm_grid(const GemmCall& c) {
  if (c.ts[0]->grid == SSS_GRID_ASYM) return gemm_bn<Q, true>(c);
  return gemm_bn<Q, false>(c);
}

}  // namespace

// the workspace that lets the call take its preferred plan (with split K
// where it helps); x16_bytes alone is enough to run it unsplit
size_t gemm_multi_workspace_bytes(const sss_qtensor_t* const* ts, int count, int64_t m) {
  const size_t x = x16_bytes(m, ts[0]->k);
  if (x == SIZE_MAX) return SIZE_MAX;
  const int64_t rt = row_tiles(ts, count);
  return x + split_bytes(rt, m, plan_gemm(rt, ts[0]->k, m, SIZE_MAX));
}
size_t gemm_workspace_bytes(const sss_qtensor_t& t, int64_t m) {
  const sss_qtensor_t* one[1] = {&t};
  return gemm_multi_workspace_bytes(one, 1, m);
}
size_t gemm_workspace_min_bytes(const sss_qtensor_t& t, int64_t m) { return x16_bytes(m, t.k); }

cudaError_t launch_gemm_multi(const sss_qtensor_t* const* ts, float* const* ys, int count,
                              const uint16_t* x, int64_t m, void* workspace, size_t ws_bytes,
                              uint32_t* status, cudaStream_t stream, bool act_q8) {
  if (count < 1 || count > kMaxGemmJobs) return cudaErrorInvalidValue;
  const int64_t k = ts[0]->k;
  __half* x16 = static_cast<__half*>(workspace);
  const int64_t rt = row_tiles(ts, count);
  const GemmPlan plan = plan_gemm(rt, k, m, ws_bytes);
  unsigned char* ws_split = static_cast<unsigned char*>(workspace) + x16_bytes(m, k);
  cudaError_t e;
  if (act_q8) {
    e = launch_act_q8_f16(x, m, k, x16, status, stream);
  } else {
    const int64_t nvec = m * k / 8;
    const int grid = static_cast<int>(std::min<int64_t>((nvec + 255) / 256,
                                                        static_cast<int64_t>(device_sm_count()) * 8));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(std::max(grid, 1)), 1, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, bf16_to_f16_kernel, x, x16, nvec);
  }
  if (e != cudaSuccess) return e;
  const GemmCall c{ts, ys, count, x16, m, status, stream, plan, ws_split};
  switch (ts[0]->q) {
    case 2: return gemm_grid<2>(c);
    case 3: return gemm_grid<3>(c);
    case 4: return gemm_grid<4>(c);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm(const sss_qtensor_t& t, const uint16_t* x, int64_t m, float* y,
                        void* workspace, size_t ws_bytes, uint32_t* status, cudaStream_t stream,
                        bool act_q8) {
  const sss_qtensor_t* one[1] = {&t};
  float* ys[1] = {y};
  return launch_gemm_multi(one, ys, 1, x, m, workspace, ws_bytes, status, stream, act_q8);
}

}  // namespace sss
