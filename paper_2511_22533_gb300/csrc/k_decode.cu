// k_decode.cu -- K10: the convolutional stand-in grid decoder O(S) of Eq. 1
// (Sec. 4.1) and the dynamic-voxel count at the anchor step (Sec. 4.2).
//
// TRELLIS's decoder is not part of the paper; this one has the shape of an
// upsampling 3-D convolution stack: 3x3x3 convolutions with zero padding and
// ReLU, C -> 16 at D^3, nearest 2x upsampling, 16 -> 8 at (2D)^3, 2x, 8 -> 1
// at (4D)^3; sub-voxel v is occupied iff its logit > 0.  Every output is
// summed in one fixed fp32 order (bias, then tap k = 0..26 with dx fastest,
// then input channel; one rounding per * and +; taps outside the grid
// skipped), so the occupancy bits are reproducible bit for bit.  The
// decoder runs twice per sample (before and after the anchor step) on a few
// hundred thousand outputs: one thread per output voxel (all output channels
// of it), weights in shared memory, no tensor cores.
#include "common.cuh"
#include "kernels.h"

namespace f3dc {

namespace {

constexpr int kDecThreads = 256;

// out[b][co][v] for v on the (din * up)^3 grid; input element (b, ci, u) at
// in + b * in_bs + ci * in_cs + u * in_vs for u on the din^3 grid.  One
// thread per output voxel computes all COUT channels, so each input value is
// loaded once for COUT products; the weights sit in shared memory as fp32.
template <int CIN, int COUT>
__global__ void __launch_bounds__(kDecThreads) k_conv3d(const float *in, size_t in_bs, size_t in_cs, size_t in_vs,
                                                       int din, int up, const uint16_t *w, const uint16_t *bias,
                                                       int relu, float *out, int B)
{
    __shared__ float sw[27][CIN][COUT];
    __shared__ float sb[COUT];
    for (int q = threadIdx.x; q < COUT * CIN * 27; q += blockDim.x) {
        const int co = q / (CIN * 27), ci = (q / 27) % CIN, k = q % 27;
        sw[k][ci][co] = bf16_bits_to_f32(w[q]);
    }
    for (int q = threadIdx.x; q < COUT; q += blockDim.x) sb[q] = bf16_bits_to_f32(bias[q]);
    __syncthreads();
    griddep_launch();
    griddep_wait();
    const int d = din * up;
    const size_t vout = (size_t)d * d * d;
    for (size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x; q < (size_t)B * vout;
         q += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(q / vout);
        const size_t v = q - (size_t)b * vout;
        const int x = (int)(v % d), y = (int)((v / d) % d), z = (int)(v / ((size_t)d * d));
        const float *ib = in + (size_t)b * in_bs;
        float acc[COUT];
#pragma unroll
        for (int co = 0; co < COUT; ++co) acc[co] = sb[co];
        for (int k = 0; k < 27; ++k) {
            const int zz = z + k / 9 - 1, yy = y + (k / 3) % 3 - 1, xx = x + k % 3 - 1;
            if (zz < 0 || zz >= d || yy < 0 || yy >= d || xx < 0 || xx >= d) continue;
            const size_t src = ((size_t)(zz / up) * din + (size_t)(yy / up)) * din + (size_t)(xx / up);
#pragma unroll
            for (int ci = 0; ci < CIN; ++ci) {
                const float xv = ib[(size_t)ci * in_cs + src * in_vs];
#pragma unroll
                for (int co = 0; co < COUT; ++co) acc[co] = __fadd_rn(acc[co], __fmul_rn(xv, sw[k][ci][co]));
            }
        }
        float *ob = out + (size_t)b * COUT * vout + v;
#pragma unroll
        for (int co = 0; co < COUT; ++co) ob[(size_t)co * vout] = relu ? (acc[co] > 0.0f ? acc[co] : 0.0f) : acc[co];
    }
}

// Last layer (8 -> 1 at (din * 2)^3) straight to occupancy bits, 32 sub-voxels
// per word (ballot of a warp's consecutive outputs); compare != 0 counts the
// bits that differ from the stored ones into dyn[b] instead of storing.
__global__ void __launch_bounds__(kDecThreads) k_conv3d_occ(const float *in, int din, const uint16_t *w,
                                                           const uint16_t *bias, uint32_t *bits, int compare,
                                                           int64_t *dyn, int B)
{
    constexpr int cin = 8, up = 2;
    __shared__ float sw[cin * 27];
    for (int q = threadIdx.x; q < cin * 27; q += blockDim.x) sw[q] = bf16_bits_to_f32(w[q]);
    __syncthreads();
    griddep_launch();
    griddep_wait();
    const int d = din * up;
    const size_t vin = (size_t)din * din * din, vout = (size_t)d * d * d;
    const int lane = threadIdx.x & 31;
    // B * vout is a multiple of 32 and so is every warp's first index, so a
    // warp's 32 outputs belong to one sample and all take the same branch
    for (size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x; q < (size_t)B * vout;
         q += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(q / vout);
        const size_t v = q - (size_t)b * vout;
        const int x = (int)(v % d), y = (int)((v / d) % d), z = (int)(v / ((size_t)d * d));
        const float *ib = in + (size_t)b * cin * vin;
        float acc = bf16_bits_to_f32(bias[0]);
        for (int k = 0; k < 27; ++k) {
            const int zz = z + k / 9 - 1, yy = y + (k / 3) % 3 - 1, xx = x + k % 3 - 1;
            if (zz < 0 || zz >= d || yy < 0 || yy >= d || xx < 0 || xx >= d) continue;
            const size_t src = ((size_t)(zz / up) * din + (size_t)(yy / up)) * din + (size_t)(xx / up);
#pragma unroll
            for (int ci = 0; ci < cin; ++ci) acc = __fadd_rn(acc, __fmul_rn(ib[(size_t)ci * vin + src], sw[ci * 27 + k]));
        }
        const uint32_t word = __ballot_sync(0xffffffffu, acc > 0.0f);
        if (lane == 0) {
            const size_t wi = q / 32;
            if (compare) {
                const int flips = __popc(word ^ bits[wi]);
                if (flips) atomicAdd(reinterpret_cast<unsigned long long *>(dyn + b), (unsigned long long)flips);
            } else {
                bits[wi] = word;
            }
        }
    }
}

int dec_grid(size_t total, int num_sms)
{
    const size_t need = (total + kDecThreads - 1) / kDecThreads;
    const size_t cap = (size_t)num_sms * 8;
    return (int)(need < cap ? (need > 0 ? need : 1) : cap);
}

}  // namespace

size_t decode_scratch_floats(int B, int D)
{
    const size_t N = (size_t)D * D * D;
    return (size_t)B * (16 * N + 8 * 8 * N);
}

cudaError_t launch_decode_conv(const DecodeArgs &a, cudaStream_t s)
{
    if (a.B < 1 || a.D < 1 || ((size_t)a.D * a.D * a.D) % 32 != 0) return cudaErrorInvalidValue;
    const int D = a.D;
    const size_t N = (size_t)D * D * D;
    float *x1 = a.scratch, *x2 = a.scratch + (size_t)a.B * 16 * N;
    // C -> 16 at D^3 from the token-major latents S [B, N, 8]
    launch_k(k_conv3d<kChannels, 16>, dim3(dec_grid((size_t)a.B * N, a.num_sms)), dim3(kDecThreads), 0, s, a.S,
             (size_t)N * kChannels, (size_t)1, (size_t)kChannels, D, 1, a.w1, a.b1, 1, x1, a.B);
    // 16 -> 8 at (2D)^3
    launch_k(k_conv3d<16, 8>, dim3(dec_grid((size_t)a.B * 8 * N, a.num_sms)), dim3(kDecThreads), 0, s,
             (const float *)x1, (size_t)16 * N, N, (size_t)1, D, 2, a.w2, a.b2, 1, x2, a.B);
    // 8 -> 1 at (4D)^3, to bits
    launch_k(k_conv3d_occ, dim3(dec_grid((size_t)a.B * 64 * N, a.num_sms)), dim3(kDecThreads), 0, s,
             (const float *)x2, 2 * D, a.w3, a.b3, a.bits, a.compare, a.dyn, a.B);
    return cudaGetLastError();
}

}  // namespace f3dc
