// Device helpers shared by the persistent forward kernels: named barriers,
// tagged cross-CTA words, bounded waits and the inner mixing loops.
#pragma once

#include "moce_mix_tile.cuh"

namespace moce {

constexpr uint32_t kSpinLimit = 1u << 20;  // polls before a wait gives up (about a second)

__device__ __forceinline__ void bar_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}
// Barrier over count threads that also returns the AND of pred over them.
__device__ __forceinline__ bool bar_and(int id, int count, bool pred) {
    int r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.s32 p, %1, 0;\n\t"
        "bar.red.and.pred q, %2, %3, p;\n\tselp.s32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((int)pred), "r"(id), "r"(count)
        : "memory");
    return r != 0;
}
__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
// Streaming 16-byte load of x that does not allocate in L1.
__device__ __forceinline__ uint4 ld_stream(const uint16_t *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// A tagged word holds an fp32 value in its low half and a tag (epoch + 1 of
// the forward that wrote it) in its high half, written by one 64-bit store,
// so a reader knows from the word itself whether the value is current.
__device__ __forceinline__ unsigned long long ld_tagged(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_tagged(unsigned long long *p, float v, uint32_t tag) {
    const unsigned long long w = ((unsigned long long)tag << 32) | __float_as_uint(v);
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}
__device__ __forceinline__ bool tag_ok(unsigned long long w, uint32_t tag) {
    return (uint32_t)(w >> 32) == tag;
}
__device__ __forceinline__ float tag_val(unsigned long long w) {
    return __uint_as_float((uint32_t)w);
}

// Records a wait that gave up: the error word makes every other wait return.
__device__ __forceinline__ void report_timeout(uint32_t *ctrl, uint32_t item) {
    atomicOr(ctrl + kCtrlError, kErrTimeout);
    atomicCAS(ctrl + kCtrlErrorItem, 0u, item + 1u);
}

// Bounded wait until the word at p carries tag; w holds the last value read.
// False when this or another wait gave up.
static __device__ bool wait_tagged(const unsigned long long *p, uint32_t tag, unsigned long long &w,
                                   uint32_t *ctrl, uint32_t item) {
    for (uint32_t it = 0; it < kSpinLimit; ++it) {
        if (tag_ok(w, tag)) return true;
        if (ld_relaxed(ctrl + kCtrlError) != 0u) return false;
        __nanosleep(it < 32 ? 64 : 256);
        w = ld_tagged(p);
    }
    report_timeout(ctrl, item);
    return false;
}

// Sets this warpgroup's registers per thread to N, from the launch's L.
// The sum over the warpgroups of a launch must stay within threads x L:
// setmaxnreg.inc waits until the registers are free.
template <int N, int L> __device__ __forceinline__ void set_role_regs() {
    static_assert(N % 8 == 0 && N >= 24 && N <= 256, "setmaxnreg count");
    if constexpr (N > L)
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(N) : "memory");
    else if constexpr (N < L)
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(N) : "memory");
}

// ---------------------------------------------------------------- mbarriers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t a) {
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(a)
                 : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t a, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(a), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait for the phase with the given parity to complete.
// try_wait suspends the warp in hardware (up to the hint) instead of
// spinning, so waiting warps leave the issue slots to the other roles.
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(a), "r"(parity), "r"(1000u)
        : "memory");
    return ok != 0;
}
static __device__ bool mbar_wait(uint32_t a, uint32_t parity, uint32_t *ctrl, uint32_t item) {
    for (uint32_t it = 0; it < kSpinLimit; ++it) {
        if (mbar_try(a, parity)) return true;
        if ((it & 15u) == 15u && ld_relaxed(ctrl + kCtrlError) != 0u) return false;
    }
    report_timeout(ctrl, item);
    return false;
}

// Release store / acquire load of a flag that CTAs of one launch exchange.
__device__ __forceinline__ void st_release(uint32_t *p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ unsigned long long ld_relaxed64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

// u / d for 0 <= u < 2^24, 1 <= d and u / d < 2^21, with inv = 1.0f / d: the float
// estimate is within one of the quotient and is corrected exactly.
__device__ __forceinline__ int fdiv(int u, int d, float inv) {
    int q = __float2int_rz(__fmul_rz((float)u, inv));
    q += (q + 1) * d <= u;
    q -= q * d > u;
    return q;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    return (uint32_t)f32_to_bf16(lo) | ((uint32_t)f32_to_bf16(hi) << 16);
}


// Table slot (uint4 units) of entries (2*i2, 2*i2+1) of expert el. The two
// lane groups of a warp mix experts 32 apart; block b of 32 experts is shifted
// by 64 * ceil(b / 2) bytes, so adjacent blocks differ by 64 bytes (their
// table reads hit different banks) and no two experts overlap.
__device__ __forceinline__ int tslot(int el, int kp, int i2) {
    return el * (kp >> 1) + ((((el >> 5) + 1) >> 1) << 2) + i2;
}
__host__ __device__ inline int tslot_count(int R, int kp) {
    return R > 0 ? (R - 1) * (kp >> 1) + (((((R - 1) >> 5) + 1) >> 1) << 2) + (kp >> 1) : 0;
}

// Weighted sum over two experts' table pairs for the lane's 8 positions;
// the two experts are interleaved for instruction-level parallelism. A table
// entry is {row offset, row offset, weight, weight} of two support positions.
__device__ __forceinline__ void mix_entries2(const unsigned char *xs, const uint4 *ta,
                                             const uint4 *tb, int npairs, uint32_t lx,
                                             float2 &a0, float2 &a1, float2 &a2, float2 &a3,
                                             float2 &b0, float2 &b1, float2 &b2, float2 &b3) {
#pragma unroll 2
    for (int i2 = 0; i2 < npairs; ++i2) {
        const uint4 ea = ta[i2];
        const uint4 eb = tb[i2];
        const uint4 va0 = lds128(xs + (ea.x ^ lx));
        const uint4 va1 = lds128(xs + (ea.y ^ lx));
        const uint4 vb0 = lds128(xs + (eb.x ^ lx));
        const uint4 vb1 = lds128(xs + (eb.y ^ lx));
        const float2 wa0 = make_float2(__uint_as_float(ea.z), __uint_as_float(ea.z));
        const float2 wa1 = make_float2(__uint_as_float(ea.w), __uint_as_float(ea.w));
        const float2 wb0 = make_float2(__uint_as_float(eb.z), __uint_as_float(eb.z));
        const float2 wb1 = make_float2(__uint_as_float(eb.w), __uint_as_float(eb.w));
        a0 = __ffma2_rn(wa0, unpack2(va0.x), a0);
        a1 = __ffma2_rn(wa0, unpack2(va0.y), a1);
        a2 = __ffma2_rn(wa0, unpack2(va0.z), a2);
        a3 = __ffma2_rn(wa0, unpack2(va0.w), a3);
        b0 = __ffma2_rn(wb0, unpack2(vb0.x), b0);
        b1 = __ffma2_rn(wb0, unpack2(vb0.y), b1);
        b2 = __ffma2_rn(wb0, unpack2(vb0.z), b2);
        b3 = __ffma2_rn(wb0, unpack2(vb0.w), b3);
        a0 = __ffma2_rn(wa1, unpack2(va1.x), a0);
        a1 = __ffma2_rn(wa1, unpack2(va1.y), a1);
        a2 = __ffma2_rn(wa1, unpack2(va1.z), a2);
        a3 = __ffma2_rn(wa1, unpack2(va1.w), a3);
        b0 = __ffma2_rn(wb1, unpack2(vb1.x), b0);
        b1 = __ffma2_rn(wb1, unpack2(vb1.y), b1);
        b2 = __ffma2_rn(wb1, unpack2(vb1.z), b2);
        b3 = __ffma2_rn(wb1, unpack2(vb1.w), b3);
    }
}

// Weighted sum over a list of table pairs for the lane's 8 positions.
__device__ __forceinline__ void mix_entries(const unsigned char *xs, const uint4 *te, int npairs,
                                            uint32_t lx, float2 &acc0, float2 &acc1, float2 &acc2,
                                            float2 &acc3) {
#pragma unroll 4
    for (int i2 = 0; i2 < npairs; ++i2) {
        const uint4 en = te[i2];
        const uint4 v0 = lds128(xs + (en.x ^ lx));
        const uint4 v1 = lds128(xs + (en.y ^ lx));
        const float wa = __uint_as_float(en.z), wb = __uint_as_float(en.w);
        const float2 w0 = make_float2(wa, wa), w1 = make_float2(wb, wb);
        acc0 = __ffma2_rn(w0, unpack2(v0.x), acc0);
        acc1 = __ffma2_rn(w0, unpack2(v0.y), acc1);
        acc2 = __ffma2_rn(w0, unpack2(v0.z), acc2);
        acc3 = __ffma2_rn(w0, unpack2(v0.w), acc3);
        acc0 = __ffma2_rn(w1, unpack2(v1.x), acc0);
        acc1 = __ffma2_rn(w1, unpack2(v1.y), acc1);
        acc2 = __ffma2_rn(w1, unpack2(v1.z), acc2);
        acc3 = __ffma2_rn(w1, unpack2(v1.w), acc3);
    }
}

// Staging unit q (chunk), j (word), cc (8-channel block) of a 16-lane tile
// (see stage_x_tile): u enumerates units so that a warp's stores are
// conflict-free.
__device__ __forceinline__ void stage_unit_coords(int u, int per_q, float inv_perq, int &q, int &j,
                                                  int &cc) {
    q = fdiv(u, per_q, inv_perq);
    const int rem = u - q * per_q;
    cc = ((rem >> 5) << 3) | (rem & 7);
    j = (rem >> 3) & 3;
}

// Stores two prefetched 8-channel vectors of positions pa and pb = pa + GS as
// eight words of the transposed tile (layout of stage_x_tile).
template <int GS>
__device__ __forceinline__ void store_unit(unsigned char *xs, int q, int j, int cc, uint4 va,
                                           uint4 vb) {
    constexpr int RB = 16 * GS;
    constexpr int FM = (GS < 8 ? GS : 8) - 1;
    unsigned char *d = xs + (size_t)(cc * 8) * RB + (((q ^ (cc & FM)) << 4) | (j << 2));
    *reinterpret_cast<uint32_t *>(d + 0 * RB) = __byte_perm(va.x, vb.x, 0x5410);
    *reinterpret_cast<uint32_t *>(d + 1 * RB) = __byte_perm(va.x, vb.x, 0x7632);
    *reinterpret_cast<uint32_t *>(d + 2 * RB) = __byte_perm(va.y, vb.y, 0x5410);
    *reinterpret_cast<uint32_t *>(d + 3 * RB) = __byte_perm(va.y, vb.y, 0x7632);
    *reinterpret_cast<uint32_t *>(d + 4 * RB) = __byte_perm(va.z, vb.z, 0x5410);
    *reinterpret_cast<uint32_t *>(d + 5 * RB) = __byte_perm(va.z, vb.z, 0x7632);
    *reinterpret_cast<uint32_t *>(d + 6 * RB) = __byte_perm(va.w, vb.w, 0x5410);
    *reinterpret_cast<uint32_t *>(d + 7 * RB) = __byte_perm(va.w, vb.w, 0x7632);
}

}  // namespace moce
