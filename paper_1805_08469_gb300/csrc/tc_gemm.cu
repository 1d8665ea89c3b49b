// Grouped TF32 products on the tcgen05 tensor cores, the accumulator in tensor memory.
//
// One CTA computes one 128 x BN tile of C[g] for group g = blockIdx.z, in k-blocks of 32
// fp32 values (128 bytes per operand row), with its warps in two roles that meet only at
// shared-memory barriers:
//   - producers (warps 0-7, 256 threads): each k-block of A (128 rows) and B (BN rows) is
//     copied from global memory with cp.async into one of kStages shared-memory stages, in
//     the 128-byte-swizzled K-major layout (the 16-byte chunk c, k = 4c .. 4c + 3, of row r
//     goes to chunk c ^ (r % 8) of the row's 128 bytes), each stage 1024-byte aligned, as
//     16-byte chunks along k.  Copies outside the operand are zero-filled.  Copies run
//     kAhead k-blocks ahead; once a thread's copies of a k-block have landed it rounds its
//     own chunks in place to TF32 (to nearest, ties away from zero: the operand values the
//     rest of the library and the oracle use; operands that are TF32 already are not
//     rounded again), makes them visible to the tensor cores' proxy and arrives on the
//     stage's `full` barrier.  A stage is refilled once its `empty` barrier says the MMAs
//     that read it have completed.
//   - MMA (warp 8, one lane): for each k-block it waits on `full`, issues four
//     tcgen05.mma.cta_group::1.kind::tf32 (K = 8 each: the descriptors' start address
//     advances 32 bytes; M = 128, N = BN, fp32 accumulation in BN columns of tensor memory
//     that warp 8 allocates), and tcgen05.commit arrives on the stage's `empty` barrier once
//     they have completed; a last commit signals `done`.
//   - epilogue (warps 0-7): warps w and w + 4 read tensor-memory lanes 32 (w % 4) .. + 31
//     (rows of the tile) with tcgen05.ld, alternate 32-column blocks each; every block goes
//     through a 32 x 33 transpose in shared memory, so that a warp stores whole row segments
//     (coalesced), after the epilogue's bias or ReLU; stored rounded to TF32 where the
//     caller asks (outputs that are only ever operands).
// Before the CTA exits, every `empty` barrier has received the arrival of its last commit
// (no arrival from the tensor cores is pending on shared memory that a later CTA may reuse)
// and warp 8 frees the tensor memory.  Every wait gives up after a bounded time: it raises a
// shared abort flag that ends both roles' loops, the CTA still drains the MMAs it issued
// (bounded) and frees its tensor memory, and the failure is reported in *status.  Every
// global access is checked against the extent of its buffer.
#include "tc_gemm.h"

#include "pdl.h"

namespace gem {
namespace tc {
namespace {

constexpr int kBM = 128;        // tile rows (the M of one MMA)
constexpr int kBK = 32;         // k per k-block: 32 fp32 = one 128-byte swizzle row
constexpr int kProducers = 256;             // warps 0-7: copies, rounding, epilogue
constexpr int kMmaWarp = kProducers / 32;   // warp 8: tensor memory and the MMAs
constexpr int kThreads = kProducers + 32;
constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s

// Per tile width and K: the stages and how many k-blocks of copies run ahead of the
// rounding (the other kStages - kAhead stages are the MMAs' slack before a refill has to
// wait).  64-wide tiles: 4 stages (96 KB, two CTAs per SM), 2 ahead for long K, 3 for short
// K (all of it in flight); 128-wide tiles: 6 stages (192 KB, one CTA per SM), 4 ahead.
template <int BN, bool DEEP>
struct Cfg {
  static constexpr int kStages = BN == 64 ? 4 : 6;
  static constexpr int kAhead = BN == 64 ? (DEEP ? 2 : 3) : 4;
  static constexpr int kATile = kBM * kBK * 4;         // bytes
  static constexpr int kBTile = BN * kBK * 4;
  static constexpr int kStage = kATile + kBTile;       // multiple of 1024
  static constexpr int kBarrierAt = kStages * kStage;  // full[], empty[], done, slot, abort
  static constexpr int kSmem = kBarrierAt + 256 + 1024; // + alignment slack
  static constexpr int kAChunks = kBM * 8 / kProducers;  // 16-byte chunks per producer
  static constexpr int kBChunks = BN * 8 / kProducers;
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

__device__ __forceinline__ void cp_async16(uint32_t dst, const float* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// TF32 value of x (round to nearest, ties away from zero; the low 13 bits cleared).
__device__ __forceinline__ float tf32_rna(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

// The 16-byte chunks a thread copies of one K-major operand tile (R rows of M or N, one
// k-block of 32 k), NCH of them, set up once so that a k-block only adds its k offset.  A
// chunk is 4 consecutive k of a row; a warp copies four 128-byte row segments; chunk c (k =
// 4c .. 4c + 3) of row r is stored at byte r * 128 + ((c ^ (r % 8)) * 16) of the tile (the
// 128-byte-swizzled K-major layout).  ok: the row lies in the operand and every element of it
// the copies can reach lies inside the operand's extent (otherwise the chunk is zero-filled,
// and reported when out of extent).
template <int R, int NCH>
struct TileCopy {
  const float* src[NCH];   // the chunk's first element at k-block 0
  uint32_t dst[NCH];       // byte offset of the chunk in the tile
  int kk[NCH];             // the chunk's first k within a k-block
  bool ok[NCH];
  bool rnd;                // the values still need rounding to TF32

  __device__ __forceinline__ void init(const Operand& o, long long goff, int tid, int row0,
                                       int rows_end, int K, bool& bad) {
    rnd = o.rounded == 0;
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      const int q = tid + kProducers * i;
      const int row = q >> 3, c = q & 7, gr = row0 + row;
      dst[i] = uint32_t(row) * 128u + (uint32_t(c ^ (row & 7)) << 4);
      kk[i] = 4 * c;
      const long long first = goff + (long long)gr * o.ld;
      const bool in = first >= 0 && first + (K - 1) < o.extent;
      const bool live = gr < rows_end;
      bad |= live && !in;
      ok[i] = live && in;
      src[i] = o.base + (ok[i] ? first + 4 * c : 0);
    }
  }

  // Copies of the k-block at k0 into the tile at shared address `tile`; zeros past K.
  __device__ __forceinline__ void issue(uint32_t tile, int k0, int K, const float* dummy) const {
    if (k0 + kBK <= K) {   // every k-block but possibly the last: whole chunks
#pragma unroll
      for (int i = 0; i < NCH; ++i) cp_async16(tile + dst[i], ok[i] ? src[i] + k0 : dummy, ok[i] ? 16 : 0);
      return;
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      const int bytes = ok[i] ? 4 * max(0, min(K - (k0 + kk[i]), 4)) : 0;
      cp_async16(tile + dst[i], bytes ? src[i] + k0 : dummy, bytes);
    }
  }

  // Round the thread's own chunks of the tile to TF32, in place: all loads first, so that
  // they overlap.
  __device__ __forceinline__ void round(uint8_t* tile) const {
    if (!rnd) return;
    float4 v[NCH];
#pragma unroll
    for (int i = 0; i < NCH; ++i) v[i] = *reinterpret_cast<const float4*>(tile + dst[i]);
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      v[i].x = tf32_rna(v[i].x);
      v[i].y = tf32_rna(v[i].y);
      v[i].z = tf32_rna(v[i].z);
      v[i].w = tf32_rna(v[i].w);
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i) *reinterpret_cast<float4*>(tile + dst[i]) = v[i];
  }
};

// Raise the CTA's abort flag with `code` (the first code stays).
__device__ __forceinline__ void raise_abort(int* flag, int code) { atomicCAS(flag, 0, code); }
__device__ __forceinline__ int aborted(const int* flag) {
  return *reinterpret_cast<const volatile int*>(flag);
}

__device__ __forceinline__ void bar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

template <int BN, bool DEEP, int EPI>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const __grid_constant__ Args p) {
  using C = Cfg<BN, DEEP>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + C::kBarrierAt);
  uint64_t* empty = full + C::kStages;
  uint64_t* done = empty + C::kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * kBM, g = blockIdx.z;

  // the accumulator: 128 lanes x BN fp32 columns of tensor memory
  if (warp == kMmaWarp) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(tmem_slot)),
                 "r"(BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (tid == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      bar_init(&full[s], kProducers);
      bar_init(&empty[s], 1);
    }
    bar_init(done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  gem::pdl_entry();   // the previous kernel's results are visible from here on

  const int nkb = (p.K + kBK - 1) / kBK;
  bool bad = false;
  int issued = 0;   // k-blocks whose MMAs and stage commit the MMA lane issued

  if (warp < kMmaWarp) {
    // ---- producers
    const long long a_goff = (p.A.by_worker ? (long long)p.workers[g] : (long long)g) * p.A.group_stride;
    const long long b_goff = (p.B.by_worker ? (long long)p.workers[g] : (long long)g) * p.B.group_stride;
    TileCopy<kBM, C::kAChunks> ca;
    TileCopy<BN, C::kBChunks> cb;
    ca.init(p.A, a_goff, tid, m0, p.M, p.K, bad);
    cb.init(p.B, b_goff, tid, n0, p.N, p.K, bad);
    constexpr int D = C::kAhead;   // k-blocks of copies in flight ahead of the rounding
    for (int kb = 0; kb < nkb + D; ++kb) {
      if (aborted(abort_flag)) break;
      // k-block kb - D: its copies have landed (kb groups committed so far, at most D - 1
      // of them still pending); rounded, fenced and handed to the MMA lane
      const int k = kb - D;
      if (k >= 0) {
        cp_async_wait<D - 1>();
        uint8_t* at = sm + (k % C::kStages) * C::kStage;
        ca.round(at);
        cb.round(at + C::kATile);
        fence_smem_to_async();
        bar_arrive(&full[k % C::kStages]);
      }
      if (kb < nkb) {
        const int s = kb % C::kStages, use = kb / C::kStages;
        // the stage's previous k-block (kb - kStages) must have been read by its MMAs
        if (use > 0 && !bar_wait(&empty[s], uint32_t(use - 1) & 1u)) {
          raise_abort(abort_flag, kWaitStage);
          break;
        }
        const uint32_t at = smem_addr(sm + s * C::kStage);
        ca.issue(at, kb * kBK, p.K, p.A.base);
        cb.issue(at + C::kATile, kb * kBK, p.K, p.B.base);
      }
      cp_async_commit();   // one group per iteration, empty ones included
    }
    cp_async_wait<0>();
  } else if (lane == 0) {
    // ---- MMA issue
    constexpr uint32_t idesc = idesc_tf32(kBM, BN);
    for (int kb = 0; kb < nkb; ++kb) {
      if (aborted(abort_flag)) break;
      const int s = kb % C::kStages;
      if (!bar_wait(&full[s], uint32_t(kb / C::kStages) & 1u)) {
        raise_abort(abort_flag, kWaitStage);
        break;
      }
      fence_after_sync();
      const uint32_t a_addr = smem_addr(sm + s * C::kStage);
      const uint32_t b_addr = a_addr + C::kATile;
#pragma unroll
      for (int kk = 0; kk < kBK / 8; ++kk)
        mma_tf32(tmem, slice_desc(a_addr, kk), slice_desc(b_addr, kk), idesc,
                 (kb | kk) != 0 ? 1u : 0u);
      commit_to(&empty[s]);
      issued = kb + 1;
    }
    // the accumulator is complete when every MMA issued so far is (also after an abort)
    commit_to(done);
  }
  __syncthreads();
  // the count of issued k-blocks, from the MMA lane to every thread
  int* issued_slot = abort_flag + 1;
  if (tid == kMmaWarp * 32) *issued_slot = issued;
  __syncthreads();
  issued = *issued_slot;

  const bool fin = __syncthreads_and(bar_wait(done, 0)) != 0;
  int err = aborted(abort_flag);
  if (!fin && !err) err = kWaitDone;
  // every stage commit has arrived before the CTA may exit: stage s received
  // ceil((issued - s) / C::kStages) of them, the last completing phase uses - 1
  if (fin) {
    for (int s = 0; s < C::kStages && s < issued; ++s) {
      const int uses = (issued - 1 - s) / C::kStages + 1;
      if (!bar_wait(&empty[s], uint32_t(uses - 1) & 1u) && !err) err = kWaitStage;
    }
  }
  fence_after_sync();

  if (fin && err == 0 && nkb > 0 && warp < kMmaWarp) {
    // Warps w, w + 4, w + 8, ... hold rows m0 + 32 (w % 4) + lane of the tile in tensor
    // memory and take the 32-column blocks in turn, kProducers / 128 apart.  Each
    // block goes through a 32 x 33 transpose in shared memory (the stages are free now), so
    // that the warp writes whole row segments: lane l stores column nb + l of each row.
    const int quad = warp & 3, first = warp >> 2;
    float* stg = reinterpret_cast<float*>(sm) + warp * (32 * 33);
    const long long c_goff = (long long)g * p.c_group_stride;
    const long long bias_goff = (EPI == kBias || EPI == kBiasRelu)
                                    ? (long long)p.workers[g] * p.bias_group_stride : 0;
    const long long mask_goff = EPI == kMask ? (long long)g * p.mask_group_stride : 0;
#pragma unroll 1
    for (int c = first; c < BN / 32; c += kProducers / 128) {
      const int nb = n0 + c * 32;
      if (nb >= p.N) break;   // the same for the whole warp
      float v[32];
      tmem_load32(tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(c * 32), v);
#pragma unroll
      for (int j = 0; j < 32; ++j) stg[lane * 33 + j] = v[j];
      __syncwarp();
      const int n = nb + lane;
      float bv = 0.f;
      if ((EPI == kBias || EPI == kBiasRelu) && n < p.N) {
        const long long bi = bias_goff + n;
        if (bi >= 0 && bi < p.bias_extent) bv = p.bias[bi];
        else bad = true;
      }
#pragma unroll 4
      for (int r = 0; r < 32; ++r) {
        const int m = m0 + quad * 32 + r;
        if (m >= p.M || n >= p.N) continue;
        float x = stg[r * 33 + lane];
        if (EPI == kBias) x = x + bv;
        if (EPI == kBiasRelu) x = fmaxf(x + bv, 0.f);
        if (EPI == kMask) {
          const long long mi = mask_goff + (long long)m * p.ldmask + n;
          float mv = 0.f;
          if (mi >= 0 && mi < p.mask_extent) mv = p.mask[mi];
          else bad = true;
          x = mv > 0.f ? x : 0.f;
        }
        const long long ci = c_goff + (long long)m * p.ldc + n;
        if (p.round_c) x = tf32_rna(x);
        if (ci >= 0 && ci < p.c_extent) p.C[ci] = x;
        else bad = true;
      }
      __syncwarp();
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
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN) : "memory");
  }
}

template <int BN, bool DEEP, int EPI>
cudaError_t launch_one(const Args& a, int groups, cudaStream_t st) {
  using C = Cfg<BN, DEEP>;
  static bool configured[64] = {};   // one attribute call per instantiation and device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(tc_gemm_kernel<BN, DEEP, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) configured[dev] = true;
  }
  dim3 grid(unsigned((a.N + BN - 1) / BN), unsigned((a.M + kBM - 1) / kBM), unsigned(groups));
  return gem::launch_pdl(tc_gemm_kernel<BN, DEEP, EPI>, grid, kThreads, size_t(C::kSmem), st, a);
}

template <int BN, bool DEEP>
cudaError_t launch_cfg(const Args& a, int groups, int epi, cudaStream_t st) {
  if (epi == kBiasRelu) return launch_one<BN, DEEP, kBiasRelu>(a, groups, st);
  if (epi == kBias) return launch_one<BN, DEEP, kBias>(a, groups, st);
  if (epi == kStore) return launch_one<BN, DEEP, kStore>(a, groups, st);
  return cudaErrorInvalidValue;
}

bool aligned16(const Operand& o) {
  return (reinterpret_cast<uintptr_t>(o.base) & 15u) == 0 && o.ld % 4 == 0 && o.group_stride % 4 == 0;
}

}  // namespace

bool supported(const Args& a, bool a_kmajor, bool b_kmajor, int epi) {
  // both operands K-major and 16-byte aligned (16-byte copies along k)
  return a_kmajor && b_kmajor && aligned16(a.A) && aligned16(a.B) &&
         (epi == kBiasRelu || epi == kBias || epi == kStore);
}

cudaError_t launch(const Args& a, int groups, bool a_kmajor, bool b_kmajor, int epi,
                   cudaStream_t stream) {
  if (groups < 1 || groups > kMaxGroups || a.M < 1 || a.N < 1 || a.K < 1 || !a.A.base ||
      !a.B.base || !a.C || !supported(a, a_kmajor, b_kmajor, epi))
    return cudaErrorInvalidValue;
  // Long K: 128-wide tiles with a deep ring once the launch has a block per SM, else
  // 64-wide.  Short K (under 8 k-blocks): 64-wide tiles, all of K in flight.
  const long long mt = (a.M + kBM - 1) / kBM;
  if (a.K >= 8 * kBK) {
    if (((a.N + 127) / 128) * mt * groups >= 152) return launch_cfg<128, true>(a, groups, epi, stream);
    return launch_cfg<64, true>(a, groups, epi, stream);
  }
  return launch_cfg<64, false>(a, groups, epi, stream);
}

}  // namespace tc
}  // namespace gem
