// Grouped TF32 products on the tcgen05 tensor cores, the accumulator in tensor memory.
//
// A persistent kernel: one CTA per SM walks the 128 x BN output tiles t = blockIdx.x,
// blockIdx.x + gridDim.x, ... of all groups (the workers of a segment), in k-blocks of 32
// fp32 values (128 bytes per operand row).  Its warps have four roles that meet only at
// shared-memory barriers, so that the copies, the MMAs and the epilogue of consecutive
// tiles overlap:
//   - TMA (warp 9, one lane): each k-block of A (128 rows) and B (BN rows) is loaded with
//     one tensor copy per operand (cp.async.bulk.tensor, a 3-D map of rows x k x group or
//     worker) into one of kStages shared-memory stages, in the 128-byte-swizzled K-major
//     layout, each stage 1024-byte aligned; the copy's bytes complete the stage's `loaded`
//     barrier.  Rows and k past the operand are filled with zeros by the copy.  A stage is
//     refilled once its `empty` barrier says the MMAs that read it have completed; the
//     k-block sequence runs on across tiles.
//   - rounding (warps 0-3), only for operands whose values are not TF32 already: warp r
//     takes the stages s = r mod 4 (so that each stage's phases are waited for by one warp,
//     in order; up to four k-blocks in flight); once the stage has loaded it rounds
//     the A and/or B tile in place to TF32 (to nearest, ties away from zero: the operand
//     values the rest of the library and the oracle use), makes its writes visible to the
//     tensor cores' proxy and arrives on the stage's `full` barrier.  Without rounding the
//     MMA lane waits on `loaded` itself, and these warps take half of the epilogue.
//   - MMA (warp 8, one lane): per tile it takes accumulator buffer i % 2 (2 x BN columns of
//     tensor memory, allocated by warp 8) once the epilogue has emptied it (`acc_empty`),
//     issues four tcgen05.mma.cta_group::1.kind::tf32 per k-block (K = 8 each: the
//     descriptors' start address advances 32 bytes; M = 128, N = BN, fp32 accumulation),
//     frees each stage with tcgen05.commit on its `empty` barrier, and signals the tile's
//     accumulator on `acc_full`.
//   - epilogue (warps 4-7, and 0-3 when nothing is rounded): the warp with q = warp % 4
//     reads tensor-memory lanes 32 q .. 32 q + 31 (rows of the tile) with tcgen05.ld, 32
//     columns at a time, and applies the bias, ReLU or mask in registers (lane = row);
//     C^T, rounded to TF32, is stored straight from the registers (lanes hold consecutive
//     rows), C goes through a 32 x 33 transpose in shared memory so that a warp stores whole
//     row segments, rounded to TF32 where the caller asks (outputs that are only ever
//     operands).  Then it releases the buffer on `acc_empty`.
// Before the CTA exits, every barrier has received the arrivals of the tensor cores' commits
// and of the tensor copies (none is pending on shared memory that a later CTA may reuse) and
// warp 8 frees the tensor memory.  Every wait gives up after a bounded time: it raises a
// shared abort flag that ends every role's loop, the CTA still drains the MMAs it issued
// (bounded) and frees its tensor memory, and the failure is reported in *status.  The tensor
// copies' maps cover exactly what supported() checked against the operands' extents; every
// other global access is checked against its buffer's extent.
#include "tc_gemm.h"

#include <cuda.h>

#include <algorithm>
#include <cstring>

#include "pdl.h"

namespace gem {
namespace tc {
namespace {

constexpr int kBM = 128;        // tile rows (the M of one MMA)
constexpr int kBK = 32;         // k per k-block: 32 fp32 = one 128-byte swizzle row
constexpr int kRounders = 128;              // warps 0-3: TF32 rounding in shared memory
constexpr int kEpilogue = 128;              // warps 4-7: the epilogue
constexpr int kMmaWarp = (kRounders + kEpilogue) / 32;   // warp 8: tensor memory, MMAs
constexpr int kTmaWarp = kMmaWarp + 1;                    // warp 9: tensor copies
constexpr int kThreads = kRounders + kEpilogue + 64;
constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s

// Per tile width: the stages of the ring (one CTA per SM: the ring takes 192 KB, the
// epilogue's transpose blocks 33 KB).
template <int BN>
struct Cfg {
  static constexpr int kStages = BN == 64 ? 8 : 6;
  static constexpr int kATile = kBM * kBK * 4;         // bytes
  static constexpr int kBTile = BN * kBK * 4;
  static constexpr int kStage = kATile + kBTile;       // multiple of 1024
  static constexpr int kEpiAt = kStages * kStage;      // 8 warps x 32 x 33 floats
  static constexpr int kBarrierAt = kEpiAt + 8 * 32 * 33 * 4;
  static constexpr int kSmem = kBarrierAt + 512 + 1024;   // barriers, slots; alignment slack
  static constexpr int kTmemCols = 2 * BN;             // two accumulators
};

// Kernel parameters: the product and the tensor maps of its operands (64-byte aligned, in
// the parameter space, where the tensor copies read them).
struct KParams {
  CUtensorMap ta, tb;
  Args p;
  int groups;
  int round_a, round_b;   // the operand's values still need rounding to TF32
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long now_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void bar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ bool bar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait until the phase of `bar` with the given parity has completed; false when kWaitNs
// (or 2^26 polls) passed first.
__device__ bool bar_wait(uint64_t* bar, uint32_t parity) {
  if (bar_test(bar, parity)) return true;
  const unsigned long long t0 = now_ns();
  for (uint32_t i = 1; i < (1u << 26); ++i) {
    if (bar_test(bar, parity)) return true;
    if ((i & 255u) == 0 && now_ns() - t0 > kWaitNs) return false;
  }
  return false;
}

__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// This thread's shared-memory writes, made visible to the async proxy (the tensor cores).
__device__ __forceinline__ void fence_smem_to_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Arrive on `bar` once every tcgen05 operation this thread issued before has completed.
__device__ __forceinline__ void commit_to(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_addr(bar))
               : "memory");
}

__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// 32 consecutive fp32 columns of tensor-memory lane (lane base of taddr + lane id), loaded
// and waited for in one statement, so no use of the values can precede the wait.
__device__ __forceinline__ void tmem_load32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, "
      "%30, %31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor of the K = 8 slice kk of a K-major operand tile in the
// 128-byte swizzle layout: start address >> 4 in bits 0-13 (the slice starts 32 kk bytes
// into the tile's 128-byte rows); leading byte offset 16 >> 4 in bits 16-29 (not used by a
// swizzled K-major layout whose slice lies inside one 128-byte row); stride byte offset
// 1024 >> 4 between 8-row groups in bits 32-45; version 1 in bit 46; base offset 0 in bits
// 49-51 (tiles start on 1024-byte boundaries); swizzle mode 2 = 128 bytes in bits 61-63.
__device__ __forceinline__ uint64_t slice_desc(uint32_t tile, int kk) {
  const uint32_t saddr = tile + 32u * uint32_t(kk);
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (static_cast<uint64_t>(16 >> 4) << 16) |
         (static_cast<uint64_t>(1024 >> 4) << 32) | (static_cast<uint64_t>(1) << 46) |
         (static_cast<uint64_t>(2) << 61);
}

// Instruction descriptor of kind::tf32: D fp32 (bits 4-5 = 1), A and B TF32 (bits 7-9 and
// 10-12 = 2), both K-major (bits 15, 16 = 0), no negation, N >> 3 in bits 17-22, M >> 4 in
// bits 24-28.
__host__ __device__ constexpr uint32_t idesc_tf32(int m, int n) {
  return (1u << 4) | (2u << 7) | (2u << 10) | (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(m >> 4) << 24);
}

__device__ __forceinline__ void report(unsigned* status, unsigned code) {
  if (status) atomicCAS(status, 0u, code);
}

// One tensor copy of the box at (x, y, z) of `map` into shared memory at `dst`; its bytes
// complete the transaction count of `bar`.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_addr(bar))
      : "memory");
}

// Arrive on `bar` and add `bytes` to the transaction count its current phase waits for.
__device__ __forceinline__ void bar_arrive_expect(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

// TF32 value of x (round to nearest, ties away from zero; the low 13 bits cleared).
__device__ __forceinline__ float tf32_rna(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

// Round `floats` consecutive values of a shared-memory tile to TF32 in place, by one warp:
// 16-byte chunks lane, lane + 32, ..., eight chunks in flight at a time (loads first, so
// that they overlap).  Explicit shared-space accesses.
template <int FLOATS>
__device__ __forceinline__ void round_tile(uint32_t tile, int lane) {
  constexpr int kChunks = FLOATS / 4;
  constexpr int kBatch = 8;
  static_assert(kChunks % (32 * kBatch) == 0, "tile not a multiple of the warp's batches");
#pragma unroll 1
  for (int c0 = 0; c0 < kChunks; c0 += 32 * kBatch) {
    float4 v[kBatch];
#pragma unroll
    for (int i = 0; i < kBatch; ++i)
      asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                   : "=f"(v[i].x), "=f"(v[i].y), "=f"(v[i].z), "=f"(v[i].w)
                   : "r"(tile + uint32_t(c0 + 32 * i + lane) * 16u));
#pragma unroll
    for (int i = 0; i < kBatch; ++i)
      asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(tile + uint32_t(c0 + 32 * i + lane) * 16u),
                   "f"(tf32_rna(v[i].x)), "f"(tf32_rna(v[i].y)), "f"(tf32_rna(v[i].z)), "f"(tf32_rna(v[i].w)));
  }
}

// Raise the CTA's abort flag with `code` (the first code stays).
__device__ __forceinline__ void raise_abort(int* flag, int code) { atomicCAS(flag, 0, code); }
__device__ __forceinline__ int aborted(const int* flag) {
  return *reinterpret_cast<const volatile int*>(flag);
}

__device__ __forceinline__ void bar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const __grid_constant__ KParams kp) {
  using C = Cfg<BN>;
  constexpr int S = C::kStages;
  const Args& p = kp.p;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  float* epi_stage = reinterpret_cast<float*>(sm + C::kEpiAt);
  uint64_t* loaded = reinterpret_cast<uint64_t*>(sm + C::kBarrierAt);
  uint64_t* full = loaded + S;
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* done = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  int* issued_slot = abort_flag + 1;   // k-blocks whose MMAs and stage commit were issued
  int* tiles_slot = issued_slot + 1;   // tiles whose accumulator commit was issued
  int* loads_slot = tiles_slot + 1;    // k-blocks whose tensor copies were issued

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nt = (p.N + BN - 1) / BN, mt = (p.M + kBM - 1) / kBM;
  const int total = nt * mt * kp.groups;
  const int my_tiles = int(blockIdx.x) < total ? (total - 1 - int(blockIdx.x)) / int(gridDim.x) + 1 : 0;
  const int nkb = (p.K + kBK - 1) / kBK;
  const long long Q = (long long)my_tiles * nkb;   // k-blocks of this CTA, across its tiles
  const bool rounding = kp.round_a || kp.round_b;
  // tile i of this CTA: group, first row, first column (columns fastest, so that
  // consecutive tiles share their A panel)
  auto tile_of = [&](int i, int& g, int& m0, int& n0) {
    const int t = int(blockIdx.x) + i * int(gridDim.x);
    n0 = (t % nt) * BN;
    const int r = t / nt;
    m0 = (r % mt) * kBM;
    g = r / mt;
  };

  if (warp == kMmaWarp) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(tmem_slot)),
                 "r"(C::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      bar_init(&loaded[s], 1);
      bar_init(&full[s], 32);   // the warp that rounds the stage
      bar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      bar_init(&acc_full[a], 1);
      bar_init(&acc_empty[a], rounding ? kEpilogue : kEpilogue + kRounders);
    }
    bar_init(done, 1);
    *abort_flag = 0;
    *issued_slot = 0;
    *tiles_slot = 0;
    *loads_slot = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  gem::pdl_entry();   // the previous kernel's results are visible from here on

  bool bad = false;

  // ---- epilogue: the warp with quad = warp % 4 holds rows m0 + 32 quad + lane of the tile
  // in tensor memory and takes the 32-column blocks c_first, c_first + c_step, ...  Per
  // block the epilogue's arithmetic runs in registers (lane = row); C^T is stored straight
  // from them (lanes hold consecutive rows: whole rows of C^T), and C goes through a 32 x 33
  // transpose in shared memory, so that lane l stores column nb + l of each row (whole row
  // segments).  Shared memory is reached through explicit shared-space loads and stores, so
  // that no access waits on a global store.  Warps 4-7 take every block; when no operand
  // needs rounding, warps 0-3 share the blocks with them (even and odd blocks).
  auto epilogue = [&](int c_first, int c_step, int warp_slot) {
    const int quad = warp & 3;
    // plain stores (the weight gradients, which the commit reads next) are kept in L2 ahead
    // of other lines (evict-last), the rest written through normally
    uint64_t keep = 0;
    if (EPI == kStore) asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep));
    const uint32_t stg = smem_addr(epi_stage + warp_slot * (32 * 33));
    for (int i = 0; i < my_tiles; ++i) {
      // warp-uniform decisions: tensor-memory loads are warp-wide
      if (__any_sync(0xffffffffu, aborted(abort_flag) != 0)) break;
      const int a = i & 1;
      if (!__all_sync(0xffffffffu, bar_wait(&acc_full[a], uint32_t(i >> 1) & 1u))) {
        raise_abort(abort_flag, kWaitDone);
        break;
      }
      fence_after_sync();
      int g, m0, n0;
      tile_of(i, g, m0, n0);
      const int m_lane = m0 + quad * 32 + lane;   // this lane's row
      const long long c_goff = (long long)g * p.c_group_stride;
      const long long bias_goff = (EPI == kBias || EPI == kBiasRelu)
                                      ? (long long)p.workers[g] * p.bias_group_stride : 0;
      const long long mask_row = EPI == kMask ? (long long)g * p.mask_group_stride + (long long)m_lane * p.ldmask : 0;
      const long long ct_goff = (long long)g * p.ct_group_stride;
#pragma unroll 1
      for (int c = c_first; c < BN / 32; c += c_step) {
        const int nb = n0 + c * 32;
        if (nb >= p.N) break;   // the same for the whole warp
        float v[32];
        tmem_load32(tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(a * BN + c * 32), v);
        if (EPI == kBias || EPI == kBiasRelu) {
          // lane l fetches bias[nb + l]; column j takes it from lane j
          const int n = nb + lane;
          float bl = 0.f;
          if (n < p.N) {
            const long long bi = bias_goff + n;
            if (bi >= 0 && bi < p.bias_extent) bl = p.bias[bi];
            else bad = true;
          }
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float bj = __shfl_sync(0xffffffffu, bl, j);
            v[j] = EPI == kBias ? v[j] + bj : fmaxf(v[j] + bj, 0.f);
          }
        }
        if (EPI == kMask && m_lane < p.M) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            if (nb + j < p.N) {
              const long long mi = mask_row + nb + j;
              float mv = 0.f;
              if (mi >= 0 && mi < p.mask_extent) mv = p.mask[mi];
              else bad = true;
              v[j] = mv > 0.f ? v[j] : 0.f;
            }
          }
        }
        if (p.round_c) {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = tf32_rna(v[j]);
        }
        // A block wholly inside the product (its 32 rows and columns) and inside the buffers'
        // extents takes the stores without per-element checks: one row pointer, advanced by
        // the leading dimension, and 32 independent stores (one epilogue warp per scheduler
        // would otherwise wait out each store's index arithmetic and branch in turn).
        const int mq = m0 + quad * 32;
        const bool whole = mq + 32 <= p.M && nb + 32 <= p.N;
        if (p.ct) {
          // C^T, rounded to TF32: row nb + j of C^T holds column nb + j of the tile
          const long long t0 = ct_goff + (long long)nb * p.ldct + mq;
          if (__all_sync(0xffffffffu, whole && t0 >= 0 && t0 + 31 * p.ldct + 31 < p.ct_extent)) {
            float* dst = p.ct + t0 + lane;
#pragma unroll
            for (int j = 0; j < 32; ++j) __stcg(dst + (long long)j * p.ldct, tf32_rna(v[j]));
          } else if (m_lane < p.M) {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              if (nb + j < p.N) {
                const long long ti = ct_goff + (long long)(nb + j) * p.ldct + m_lane;
                if (ti >= 0 && ti < p.ct_extent) __stcg(p.ct + ti, tf32_rna(v[j]));
                else bad = true;
              }
            }
          }
        }
#pragma unroll
        for (int j = 0; j < 32; ++j)
          asm volatile("st.shared.f32 [%0], %1;" ::"r"(stg + uint32_t(lane * 33 + j) * 4u), "f"(v[j]));
        __syncwarp();
        float col[32];
#pragma unroll
        for (int r = 0; r < 32; ++r)
          asm volatile("ld.shared.f32 %0, [%1];" : "=f"(col[r]) : "r"(stg + uint32_t(r * 33 + lane) * 4u));
        const int n = nb + lane;
        const long long c0 = c_goff + (long long)mq * p.ldc + nb;
        if (__all_sync(0xffffffffu, whole && c0 >= 0 && c0 + 31 * p.ldc + 31 < p.c_extent)) {
          float* dst = p.C + c0 + lane;
#pragma unroll
          for (int r = 0; r < 32; ++r) {
            if (EPI == kStore)
              asm volatile("st.global.L2::cache_hint.f32 [%0], %1, %2;" ::"l"(dst + (long long)r * p.ldc),
                           "f"(col[r]), "l"(keep)
                           : "memory");
            else
              __stcg(dst + (long long)r * p.ldc, col[r]);
          }
        } else if (n < p.N) {
#pragma unroll
          for (int r = 0; r < 32; ++r) {
            const int m = mq + r;
            if (m < p.M) {
              const long long ci = c_goff + (long long)m * p.ldc + n;
              if (ci >= 0 && ci < p.c_extent) __stcg(p.C + ci, col[r]);
              else bad = true;
            }
          }
        }
        __syncwarp();
      }
      // the accumulator is read (tensor-memory loads waited for): hand it back
      fence_before_sync();
      bar_arrive(&acc_empty[a]);
    }
    };

  if (warp == kTmaWarp) {
    // ---- tensor copies (one lane): k-block q is k-block q % nkb of tile q / nkb
    if (lane == 0) {
      int za = 0, zb = 0, m0 = 0, n0 = 0;
      long long q = 0;
      for (; q < Q; ++q) {
        if (aborted(abort_flag)) break;
        const int s = int(q % S);
        const long long use = q / S;
        // the stage's previous k-block (q - kStages) must have been read by its MMAs
        if (use > 0 && !bar_wait(&empty[s], uint32_t(use - 1) & 1u)) {
          raise_abort(abort_flag, kWaitStage);
          break;
        }
        const int kb = int(q % nkb);
        if (kb == 0) {
          int g;
          tile_of(int(q / nkb), g, m0, n0);
          za = p.A.by_worker ? p.workers[g] : g;
          zb = p.B.by_worker ? p.workers[g] : g;
        }
        const uint32_t at = smem_addr(sm + s * C::kStage);
        bar_arrive_expect(&loaded[s], uint32_t(C::kStage));
        tma_load_3d(at, &kp.ta, kb * kBK, m0, za, &loaded[s]);
        tma_load_3d(at + C::kATile, &kp.tb, kb * kBK, n0, zb, &loaded[s]);
      }
      *loads_slot = int(q);
    }
  } else if (warp < kRounders / 32) {
    // ---- rounding of the operands that are not TF32 yet, else half of the epilogue
    if (!rounding) {
      epilogue(0, 2, warp);   // staging buffers 0-3 (the epilogue warps use 4-7)
    } else {
      for (long long q = 0; q < Q; ++q) {
        const int s = int(q % S);
        if (s % (kRounders / 32) != warp) continue;
        if (aborted(abort_flag)) break;
        if (!__all_sync(0xffffffffu, bar_wait(&loaded[s], uint32_t(q / S) & 1u))) {
          raise_abort(abort_flag, kWaitStage);
          break;
        }
        const uint32_t at = smem_addr(sm + s * C::kStage);
        if (kp.round_a) round_tile<kBM * kBK>(at, lane);
        if (kp.round_b) round_tile<BN * kBK>(at + C::kATile, lane);
        fence_smem_to_async();
        bar_arrive(&full[s]);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---- MMA issue (one lane)
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_tf32(kBM, BN);
      uint64_t* ready = rounding ? full : loaded;
      long long q = 0;
      int issued = 0, tiles = 0;
      for (int i = 0; i < my_tiles; ++i) {
        if (aborted(abort_flag)) break;
        const int a = i & 1, ua = i >> 1;
        // the accumulator's previous tile (i - 2) has been read by the epilogue
        if (ua > 0 && !bar_wait(&acc_empty[a], uint32_t(ua - 1) & 1u)) {
          raise_abort(abort_flag, kWaitStage);
          break;
        }
        fence_after_sync();
        const uint32_t d = tmem + uint32_t(a * BN);
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb, ++q) {
          const int s = int(q % S);
          if (aborted(abort_flag) || !bar_wait(&ready[s], uint32_t(q / S) & 1u)) {
            raise_abort(abort_flag, kWaitStage);
            ok = false;
            break;
          }
          fence_after_sync();
          const uint32_t a_addr = smem_addr(sm + s * C::kStage);
          const uint32_t b_addr = a_addr + C::kATile;
#pragma unroll
          for (int kk = 0; kk < kBK / 8; ++kk)
            mma_tf32(d, slice_desc(a_addr, kk), slice_desc(b_addr, kk), idesc, (kb | kk) != 0 ? 1u : 0u);
          commit_to(&empty[s]);
          issued = int(q) + 1;
        }
        if (!ok) break;
        commit_to(&acc_full[a]);
        tiles = i + 1;
      }
      // every MMA issued so far has completed once `done` does (also after an abort)
      commit_to(done);
      *issued_slot = issued;
      *tiles_slot = tiles;
    }
  } else {
    epilogue(rounding ? 0 : 1, rounding ? 1 : 2, warp);
  }

  __syncthreads();
  const int issued = *issued_slot, tiles = *tiles_slot, loads = *loads_slot;
  const bool fin = __syncthreads_and(bar_wait(done, 0)) != 0;
  int err = aborted(abort_flag);
  if (!fin && !err) err = kWaitDone;
  if (fin) {
    // every asynchronous arrival has landed before the CTA may exit: stage s received
    // ceil((n - s) / S) of n copies and n' MMA commits, accumulator a ceil((tiles - a) / 2)
    // tile commits; the last completing phase of each is uses - 1
    for (int s = 0; s < S && s < loads; ++s) {
      const int uses = (loads - 1 - s) / S + 1;
      if (!bar_wait(&loaded[s], uint32_t(uses - 1) & 1u) && !err) err = kWaitStage;
    }
    for (int s = 0; s < S && s < issued; ++s) {
      const int uses = (issued - 1 - s) / S + 1;
      if (!bar_wait(&empty[s], uint32_t(uses - 1) & 1u) && !err) err = kWaitStage;
    }
    for (int a = 0; a < 2 && a < tiles; ++a) {
      const int uses = (tiles - 1 - a) / 2 + 1;
      if (!bar_wait(&acc_full[a], uint32_t(uses - 1) & 1u) && !err) err = kWaitDone;
    }
  }
  if (err) {
    if (tid == 0) report(p.status, unsigned(err));
  } else if (bad) {
    report(p.status, kOutOfRange);
  }

  fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::kTmemCols)
                 : "memory");
  }
}

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                 CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                 CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, looked up once (the library links only the runtime).
EncodeTiled encoder() {
  static EncodeTiled fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    EncodeTiled r = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      r = reinterpret_cast<EncodeTiled>(f);
    cudaGetLastError();
    return r;
  }();
  return fn;
}

// Planes (groups or workers) an operand's copies address: the groups, or every worker up to
// the largest one named.
long long planes(const Operand& o, const Args& a, int groups) {
  if (!o.by_worker) return groups;
  int w = 0;
  for (int g = 0; g < groups; ++g) w = std::max(w, a.workers[g]);
  return (long long)w + 1;
}

// Whether every element the operand's map can address, rows x K x planes, lies inside its
// extent.
bool within(const Operand& o, long long rows, int K, long long zc) {
  if (rows < 1 || K < 1 || zc < 1 || o.ld < K || o.extent < 1) return false;
  if (zc > 1 && o.group_stride < 1) return false;
  const long long last = (zc - 1) * o.group_stride + (rows - 1) * o.ld + (K - 1);
  return last < o.extent;
}

// A 3-D map of the operand: k (innermost, K), rows, planes; boxes of 32 k x box_rows rows,
// 128-byte swizzle, zeros outside.
cudaError_t encode(CUtensorMap* map, const Operand& o, long long rows, int K, long long zc, int box_rows) {
  EncodeTiled fn = encoder();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[3] = {cuuint64_t(K), cuuint64_t(rows), cuuint64_t(zc)};
  const long long plane = zc > 1 ? o.group_stride : rows * o.ld;
  const cuuint64_t strides[2] = {cuuint64_t(o.ld) * 4u, cuuint64_t((plane + 3) / 4 * 4) * 4u};
  const cuuint32_t box[3] = {cuuint32_t(kBK), cuuint32_t(box_rows), 1u};
  const cuuint32_t estr[3] = {1u, 1u, 1u};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3u, const_cast<float*>(o.base), dims, strides,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int BN, int EPI>
cudaError_t launch_one(const Args& a, int groups, cudaStream_t st) {
  using C = Cfg<BN>;
  static bool configured[64] = {};   // one attribute call per instantiation and device
  static int sms[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  const bool cached = dev >= 0 && dev < 64 && configured[dev];
  int sm_count = cached ? sms[dev] : 0;
  if (!cached) {
    cudaError_t e = cudaFuncSetAttribute(tc_gemm_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sm_count, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) {
      sms[dev] = sm_count;
      configured[dev] = true;
    }
  }
  KParams kp;
  std::memset(&kp, 0, sizeof(kp));
  kp.p = a;
  kp.groups = groups;
  kp.round_a = a.A.rounded ? 0 : 1;
  kp.round_b = a.B.rounded ? 0 : 1;
  cudaError_t e = encode(&kp.ta, a.A, a.M, a.K, planes(a.A, a, groups), kBM);
  if (e == cudaSuccess) e = encode(&kp.tb, a.B, a.N, a.K, planes(a.B, a, groups), BN);
  if (e != cudaSuccess) return e;
  const long long tiles = (long long)((a.N + BN - 1) / BN) * ((a.M + kBM - 1) / kBM) * groups;
  if (tiles > (1ll << 30)) return cudaErrorInvalidValue;
  const int grid = int(tiles < sm_count ? tiles : sm_count);   // one CTA per SM, persistent
  return gem::launch_pdl(tc_gemm_kernel<BN, EPI>, dim3(unsigned(grid)), kThreads, size_t(C::kSmem), st, kp);
}

template <int BN>
cudaError_t launch_cfg(const Args& a, int groups, int epi, cudaStream_t st) {
  if (epi == kBiasRelu) return launch_one<BN, kBiasRelu>(a, groups, st);
  if (epi == kBias) return launch_one<BN, kBias>(a, groups, st);
  if (epi == kStore) return launch_one<BN, kStore>(a, groups, st);
  if (epi == kMask) return launch_one<BN, kMask>(a, groups, st);
  return cudaErrorInvalidValue;
}

bool aligned16(const Operand& o) {
  return (reinterpret_cast<uintptr_t>(o.base) & 15u) == 0 && o.ld % 4 == 0 && o.group_stride % 4 == 0;
}

}  // namespace

bool supported(const Args& a, bool a_kmajor, bool b_kmajor, int epi, int groups) {
  // both operands K-major, 16-byte aligned (the tensor copies' base and strides), and every
  // element their maps address inside the operand's extent
  return a_kmajor && b_kmajor && aligned16(a.A) && aligned16(a.B) && groups >= 1 &&
         groups <= kMaxGroups && within(a.A, a.M, a.K, planes(a.A, a, groups)) &&
         within(a.B, a.N, a.K, planes(a.B, a, groups)) &&
         (epi == kBiasRelu || epi == kBias || epi == kStore || epi == kMask);
}

cudaError_t launch(const Args& a, int groups, bool a_kmajor, bool b_kmajor, int epi,
                   cudaStream_t stream) {
  if (groups < 1 || groups > kMaxGroups || a.M < 1 || a.N < 1 || a.K < 1 || !a.A.base ||
      !a.B.base || !a.C || !supported(a, a_kmajor, b_kmajor, epi, groups))
    return cudaErrorInvalidValue;
  // 128-wide tiles when they still give every SM a tile (a k-block then feeds twice the MMA
  // work for 4/3 of the bytes); otherwise 64-wide, which spreads a product with few tiles
  // (a 128-row minibatch panel per worker) over more SMs: its weights come from DRAM, and
  // more SMs pulling them finish sooner than fewer copying fewer bytes each (measured: the
  // forward products of a 13-worker segment 29.7 us 64-wide, 36 us 128-wide)
  const long long tiles128 = (long long)((a.N + 127) / 128) * ((a.M + kBM - 1) / kBM) * groups;
  if (tiles128 >= 152) return launch_cfg<128>(a, groups, epi, stream);
  return launch_cfg<64>(a, groups, epi, stream);
}

}  // namespace tc
}  // namespace gem
