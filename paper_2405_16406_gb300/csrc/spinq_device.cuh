// spinq_device.cuh -- device helpers shared by the sm_103a kernels of the
// rotated W4A4 library: inline-PTX wrappers for warp MMA, mbarriers, TMA and
// tcgen05, and the fp32 -> 4-bit code packing used by every quantizer.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

namespace spinq {

// ---------------------------------------------------------------------------
// Warp-level fp16 MMA (m16n8k16, fp32 accumulate).  Used for the Hadamard
// stages that read the raw fp16 input: the matrix entries are +-1 (exact in
// fp16) and the products are accumulated in fp32.
// A fragment: a[0] = (row g, k 2c..2c+1), a[1] = (row g+8, k 2c..2c+1),
//             a[2] = (row g, k 2c+8..2c+9), a[3] = (row g+8, k 2c+8..2c+9)
// B fragment: b[0] = (k 2c..2c+1, n g), b[1] = (k 2c+8..2c+9, n g)
// D fragment: d[0..1] = (row g, n 2c..2c+1), d[2..3] = (row g+8, n 2c..2c+1)
// with g = lane / 4, c = lane % 4.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mma_16816_f16_f32(float d[4], const uint32_t a[4], uint32_t b0,
                                                  uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%10,%11,%12,%13};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f), "f"(0.f),
        "f"(0.f), "f"(0.f));
}

// Same MMA accumulating into d (C = D).
__device__ __forceinline__ void mma_16816_f16_f32_acc(float d[4], const uint32_t a[4], uint32_t b0,
                                                      uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Four 8x8 b16 matrices from shared memory, transposed: lane l supplies the
// address of row (l % 8) of matrix (l / 8); register q then holds, in lane
// (g, c), elements (row 2c, col g) and (row 2c + 1, col g) of matrix q.
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t r[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ uint32_t pack_half2_bits(float lo, float hi) {
  __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// ---------------------------------------------------------------------------
// Packed fp32 pairs.  sm_100-family SMs execute add/sub/fma on two fp32 lanes
// held in one 64-bit register pair (PTX add/sub/fma.rn.f32x2) as a single
// instruction; each lane is rounded exactly like the scalar operation, so the
// results are bit-identical to scalar FADD/FFMA code.  The Hadamard butterflies
// and the quantizer's scale step run on these pairs.
// ---------------------------------------------------------------------------
struct F2 {
  unsigned long long u;
};

__device__ __forceinline__ F2 f2_make(float lo, float hi) {
  F2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r.u) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(F2 x, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(x.u));
}
__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
  F2 r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r.u) : "l"(a.u), "l"(b.u));
  return r;
}
__device__ __forceinline__ F2 f2_sub(F2 a, F2 b) {
  F2 r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r.u) : "l"(a.u), "l"(b.u));
  return r;
}
__device__ __forceinline__ F2 f2_fma(F2 a, F2 b, F2 c) {
  F2 r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r.u) : "l"(a.u), "l"(b.u), "l"(c.u));
  return r;
}
__device__ __forceinline__ F2 f2_mul(F2 a, F2 b) {
  F2 r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r.u) : "l"(a.u), "l"(b.u));
  return r;
}
// the pair (lo, hi) from two 32-bit registers holding fp32 bits
__device__ __forceinline__ F2 f2_from_bits(uint32_t lo, uint32_t hi) {
  F2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r.u) : "r"(lo), "r"(hi));
  return r;
}
// radix-2 butterfly on two pairs: (a, b) <- (a + b, a - b), lane by lane
__device__ __forceinline__ void f2_bfly(F2& a, F2& b) {
  const F2 s = f2_add(a, b);
  b = f2_sub(a, b);
  a = s;
}
// butterfly between the two lanes of one pair: (lo, hi) <- (lo + hi, lo - hi)
__device__ __forceinline__ void f2_bfly_inner(F2& a) {
  float lo, hi;
  f2_split(a, lo, hi);
  a = f2_make(lo + hi, lo - hi);
}

// Accumulating form of mma_16816_f16_f32_pairs (C = D).
__device__ __forceinline__ void mma_16816_f16_f32_pairs_acc(F2& d01, F2& d23, const uint32_t a[4], uint32_t b0,
                                                            uint32_t b1) {
  asm volatile(
      "{\n\t.reg .f32 e0, e1, e2, e3;\n\t"
      "mov.b64 {e0, e1}, %0;\n\tmov.b64 {e2, e3}, %1;\n\t"
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {e0,e1,e2,e3}, {%2,%3,%4,%5}, {%6,%7}, "
      "{e0,e1,e2,e3};\n\t"
      "mov.b64 %0, {e0, e1};\n\tmov.b64 %1, {e2, e3};\n\t}\n"
      : "+l"(d01.u), "+l"(d23.u)
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// m16n8k16 MMA whose D fragment comes back as two pairs: d01 = (d[0], d[1])
// (row g) and d23 = (d[2], d[3]) (row g + 8).
__device__ __forceinline__ void mma_16816_f16_f32_pairs(F2& d01, F2& d23, const uint32_t a[4], uint32_t b0,
                                                        uint32_t b1) {
  asm volatile(
      "{\n\t.reg .f32 e0, e1, e2, e3;\n\t"
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {e0,e1,e2,e3}, {%2,%3,%4,%5}, {%6,%7}, "
      "{%8,%8,%8,%8};\n\t"
      "mov.b64 %0, {e0, e1};\n\tmov.b64 %1, {e2, e3};\n\t}\n"
      : "=l"(d01.u), "=l"(d23.u)
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f));
}

// 1.5 * 2^23: adding it to |v| < 2^22 leaves round-half-to-even(v) in the low
// mantissa bits (the FADD rounds to nearest even), so the low nibble of the
// sum's bit pattern is the two's complement 4-bit code of rint(v).
constexpr float kRoundMagic = 12582912.0f;

__device__ __forceinline__ uint32_t round_bits(float v) {
  return __float_as_uint(v + kRoundMagic);
}

// Pack the low nibbles of eight round_bits() words: element e -> nibble e
// (even index in the low nibble of each byte).
__device__ __forceinline__ uint32_t pack8_nibbles(const uint32_t r[8]) {
  const uint32_t t02 = __byte_perm(r[0], r[2], 0x0040);
  const uint32_t t46 = __byte_perm(r[4], r[6], 0x0040);
  const uint32_t t13 = __byte_perm(r[1], r[3], 0x0040);
  const uint32_t t57 = __byte_perm(r[5], r[7], 0x0040);
  const uint32_t ev = __byte_perm(t02, t46, 0x5410);  // bytes: r0 r2 r4 r6
  const uint32_t od = __byte_perm(t13, t57, 0x5410);  // bytes: r1 r3 r5 r7
  return (ev & 0x0F0F0F0Fu) | ((od << 4) & 0xF0F0F0F0u);
}

// Two / four round_bits() words -> one byte / 16 bits of nibbles (first
// element in the low nibble).
__device__ __forceinline__ uint32_t pack2_nibbles(uint32_t r0, uint32_t r1) {
  return (r0 & 0x0Fu) | ((r1 << 4) & 0xF0u);
}
__device__ __forceinline__ uint32_t pack4_nibbles(uint32_t r0, uint32_t r1, uint32_t r2, uint32_t r3) {
  return __byte_perm(pack2_nibbles(r0, r1), pack2_nibbles(r2, r3), 0x0040);
}

// ---------------------------------------------------------------------------
// mbarrier (shared::cta) with bounded waits
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, "
      "0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;\n" : "=l"(t));
  return t;
}

// Waits for the phase of `bar` with `parity`, sleeping between polls (32 ns
// doubling to 1 us) so that waiting warps leave the issue slots to the warps
// that work.  Returns false, and raises *abort_flag, after `limit_ns` of wall
// time; returns false at once when *abort_flag is already up.
__device__ __forceinline__ bool mbar_wait_backoff(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  uint32_t ns = 32;
  while (true) {
    __nanosleep(ns);
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) {
      *abort_flag = 1;
      return false;
    }
    if (ns < 1024) ns <<= 1;
  }
}

// try_wait with a suspend-time hint: the thread sleeps in hardware until the
// phase completes (it wakes at once then) or about `hint_ns` have passed.
__device__ __forceinline__ bool mbar_try_wait_hint(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, "
      "0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

// Waits for the phase of `bar` with `parity` suspended in hardware (woken by
// the phase's completion), checking the abort flag and the time limit every
// ~20 us.  Returns false, and raises *abort_flag, after `limit_ns` of wall
// time; returns false when *abort_flag is up after a wake-up.
__device__ __forceinline__ bool mbar_wait_suspend(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait_hint(bar, parity, 20000u)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) {
      *abort_flag = 1;
      return false;
    }
  }
}

// Waits until the phase with `parity` has completed.  Gives up after
// `limit_ns` nanoseconds of wall time and returns false.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

// atomic add on a shared-memory word (the shared-space form, not a generic
// atomic); returns the old value
__device__ __forceinline__ uint32_t atom_add_shared(const void* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.shared::cta.add.u32 %0, [%1], %2;" : "=r"(old) : "r"(smem_u32(p)), "r"(v) : "memory");
  return old;
}

// Returns only once the loads that produced w[] have completed.  The XOR of
// one register of each vector cannot issue before those loads are done, and
// it feeds a predicated store to a scratch word (which practically never
// fires and is harmless when it does), so the assembler cannot drop it; the
// store is ordered before the caller's __syncwarp and mbarrier arrive.  This
// lets a warp release a shared-memory stage right after reading it without
// the arrive overtaking the loads (an arrive issued right after the loads can
// be seen before they have read shared memory, and a refill of the stage
// would then race them).
template <int N>
__device__ __forceinline__ void wait_loaded(const uint4 (&w)[N], volatile uint32_t* scratch) {
  uint32_t acc = 0x2545F491u;
#pragma unroll
  for (int j = 0; j < N; ++j) acc ^= w[j].x;
  if (acc == 0x9E3779B9u) *scratch = acc;
}

// Programmatic dependent launch.  Every kernel of the library is launched so
// that it may start while the kernel before it in the stream is finishing;
// each thread runs pdl_wait() after its shared-memory prologue and before its
// first global-memory access (read or write): it returns once the preceding
// grid has completed and its writes are visible (at once when there is no
// such grid).  pdl_trigger() lets the next kernel be scheduled once every CTA
// of this grid has reached it (grids are sized to be resident at once, so
// the next kernel's CTAs only take SM resources this grid leaves free).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;\n" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}

// ---------------------------------------------------------------------------
// TMA (tiled tensor copy, global -> shared, completion on an mbarrier)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(void* smem_dst, const void* tmap, uint64_t* bar,
                                            int32_t x, int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
      "%3}], [%4];\n" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tma_load_4d(void* smem_dst, const void* tmap, uint64_t* bar, int32_t c0,
                                            int32_t c1, int32_t c2, int32_t c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
      "%3, %4, %5}], [%6];\n" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tma_load_5d(void* smem_dst, const void* tmap, uint64_t* bar, int32_t c0,
                                            int32_t c1, int32_t c2, int32_t c3, int32_t c4) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
      "%3, %4, %5, %6}], [%7];\n" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(smem_u32(bar))
      : "memory");
}

// Bulk (non-tensor) copy global -> shared, completion on an mbarrier.  Both
// addresses 16-byte aligned, `bytes` a multiple of 16.
__device__ __forceinline__ void bulk_load(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(gsrc)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// TMA tiled store shared -> global in a bulk group; box at (x, y), elements
// outside the tensor are not written.
__device__ __forceinline__ void tma_store_2d(const void* tmap, const void* smem_src, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];\n" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(x), "r"(y), "r"(smem_u32(smem_src))
               : "memory");
}
__device__ __forceinline__ void bulk_commit_group() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }
// wait until at most N bulk groups of this thread still read shared memory
template <int N>
__device__ __forceinline__ void bulk_wait_group_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;\n" ::"n"(N) : "memory");
}
// wait until at most N bulk groups of this thread are still in flight
template <int N>
__device__ __forceinline__ void bulk_wait_group() {
  asm volatile("cp.async.bulk.wait_group %0;\n" ::"n"(N) : "memory");
}

__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05 (5th-generation tensor core, accumulators in tensor memory)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* smem_result, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                   smem_u32(smem_result)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, 8-bit floating point operands (kind::f8f6f4).
__device__ __forceinline__ void tc_mma_f8f6f4(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` once every tcgen05 operation issued so far by this thread
// has completed.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
          smem_u32(bar))
      : "memory");
}

// ---------------------------------------------------------------------------
// Thread-block clusters of two CTAs (an SM pair) and the cta_group::2 forms
// of the tcgen05 instructions, with which one thread of the pair issues MMAs
// that span both SMs (M = 256: each CTA holds 128 rows of A, half of B and
// 128 lanes of the accumulator, at the same shared/tensor memory addresses).
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t local_addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(local_addr), "r"(rank));
  return r;
}

// Arrive on an mbarrier of another CTA of the cluster, given by its cluster
// address (release semantics as for a local arrive).
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];\n" ::"r"(cluster_addr) : "memory");
}

__device__ __forceinline__ void st_shared_cluster_u32(uint32_t cluster_addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;\n" ::"r"(cluster_addr), "r"(v) : "memory");
}

// Every thread of both CTAs (release / acquire).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}

// One warp in each CTA of the pair, together.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* smem_result, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                   smem_u32(smem_result)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// Pair MMA (M = 256) issued by one thread for both CTAs.
__device__ __forceinline__ void tc_mma_pair_f8f6f4(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                   uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on the mbarrier at `bar`'s offset in every CTA of `cta_mask` once
// the pair MMAs issued so far by this thread have completed.
__device__ __forceinline__ void tc_commit_pair_mc(uint64_t* bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n" ::"r"(
          smem_u32(bar)),
      "h"(cta_mask)
      : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns from tensor memory.
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t r[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%"
      "15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

// 32 lanes x 16 consecutive 32-bit columns from tensor memory.
__device__ __forceinline__ void tmem_ld_32x32b_x16(uint32_t taddr, uint32_t r[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, "
      "[%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

// tcgen05.ld writes its destination registers asynchronously: they hold the
// data only after tcgen05.wait::ld.  Passing them through the wait as
// read-write operands makes every later use depend on it, so the compiler
// cannot schedule a use between the load and the wait.
__device__ __forceinline__ void tmem_ld_wait(uint32_t r[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;\n"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15])
               :
               : "memory");
}

// Shared-memory matrix descriptor for a K-major operand tile stored with the
// 128-byte swizzle: rows of 128 bytes, 8-row groups 1024 bytes apart, the
// 16-byte chunk c of row r stored at chunk c ^ (r % 8).  The tile base must be
// 1024-byte aligned; `addr` may point 32*k bytes into the row for the k-th
// 32-element slice.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFF);        // start address
  d |= (uint64_t)1 << 16;                        // leading byte offset (unused for SW128 K-major)
  d |= (uint64_t)(1024 >> 4) << 32;              // stride byte offset: 8 rows * 128 B
  d |= (uint64_t)1 << 46;                        // descriptor version (sm_100 family)
  d |= (uint64_t)2 << 61;                        // layout: 128-byte swizzle
  return d;
}

// Shared-memory matrix descriptor for an MN-major operand stored with the
// 128-byte swizzle: 64-element atoms along M/N, each 8 K-rows of 128 bytes
// (chunk c of row r at chunk c ^ (r % 8)); `lbo` bytes between atoms along
// M/N, `sbo` bytes between 8-row groups along K.  Base 1024-byte aligned.
__device__ __forceinline__ uint64_t umma_desc_sw128_mn(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFF);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// D[tmem] (+)= A[smem] * B[smem], 16-bit floating point operands (kind::f16).
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Instruction descriptor for kind::f16, FP16 x FP16 -> F32, A K-major, B
// MN-major (bit 16).
__host__ __device__ constexpr uint32_t umma_idesc_f16_f32_bmn(int M, int N) {
  return (1u << 4)                          // D format: F32
         | (0u << 7)                        // A format: F16
         | (0u << 10)                       // B format: F16
         | (1u << 16)                       // B MN-major
         | ((uint32_t)(N >> 3) << 17)       // N / 8
         | ((uint32_t)(M >> 4) << 24);      // M / 16
}

// Instruction descriptor for kind::f8f6f4, E4M3 x E4M3 -> F32, both K-major.
__host__ __device__ constexpr uint32_t umma_idesc_e4m3_f32(int M, int N) {
  return (1u << 4)                          // D format: F32
         | (0u << 7)                        // A format: E4M3
         | (0u << 10)                       // B format: E4M3
         | ((uint32_t)(N >> 3) << 17)       // N / 8
         | ((uint32_t)(M >> 4) << 24);      // M / 16
}

}  // namespace spinq
