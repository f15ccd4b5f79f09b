/* Test helper (compiled by tests/test_float_identities.py): checks that x / d, correctly rounded,
 * equals q + (x - q d) r with r = RN(1/d) and q = RN(x r), each step rounded once (fmaf), for every
 * 24-bit numerator significand against the given divisor significands, and for random pairs of an
 * integer numerator (|x| < 2^31) and a divisor in [2^-60, 2^60]; and, for the softmax's quotients
 * E / sum, for random numerators in [2^-100, 1] against divisors in [1, 2^24]. Prints the number of
 * pairs checked and of mismatches. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

static float from_bits(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }
static uint32_t bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }

static float div_by_recip(float x, float d, float r)
{
    float q = x * r;
    float e = fmaf(-q, d, x);
    return fmaf(e, r, q);
}

static uint64_t st = 0x9E3779B97F4A7C15ull;
static uint64_t next(void) { st ^= st << 13; st ^= st >> 7; st ^= st << 17; return st; }

int main(int argc, char **argv)
{
    long bad = 0, n = 0;
    int ndiv = argc > 1 ? atoi(argv[1]) : 64;
    long nrand = argc > 2 ? atol(argv[2]) : 10000000;
    for (int k = 0; k < ndiv; ++k) {
        uint32_t m;
        if (k < 8) m = 0x7FFFFFu - (uint32_t)k;           /* significands of all ones and neighbours */
        else if (k < 16) m = (uint32_t)(k - 8);           /* powers of two and neighbours */
        else m = (uint32_t)(next() & 0x7FFFFFu);
        float d = from_bits((127u << 23) | m);
        float r = 1.0f / d;
        for (uint32_t a = 1u << 23; a < (1u << 24); ++a) {
            float x = (float)a;
            if (bits(div_by_recip(x, d, r)) != bits(x / d)) ++bad;
            ++n;
        }
    }
    for (long i = 0; i < nrand; ++i) {
        uint64_t u = next();
        int e = (int)(u % 121) - 60;
        float d = from_bits((uint32_t)(e + 127) << 23 | (uint32_t)((u >> 8) & 0x7FFFFFu));
        int len = 1 + (int)((u >> 32) % 31);
        long long xi = (long long)((u >> 33) & ((1ull << len) - 1));
        if (u >> 63) xi = -xi;
        float x = (float)xi;
        float r = 1.0f / d;
        if (bits(div_by_recip(x, d, r)) != bits(x / d)) ++bad;
        ++n;
    }
    long nsoft = argc > 3 ? atol(argv[3]) : 0;
    for (long i = 0; i < nsoft; ++i) {
        uint64_t u = next();
        int ex = -(int)(u % 101);                         /* numerator exponent -100 .. 0 */
        uint32_t mx = (uint32_t)((u >> 8) & 0x7FFFFFu);
        float x = ex == 0 ? 1.0f : from_bits((uint32_t)(ex + 127) << 23 | mx);
        int ed = (int)((u >> 32) % 25);                   /* divisor exponent 0 .. 24 */
        uint32_t md = (uint32_t)((u >> 40) & 0x7FFFFFu);
        if ((u & 0xF) == 0) md = 0x7FFFFFu;               /* all-ones significands now and then */
        float d = from_bits((uint32_t)(ed + 127) << 23 | md);
        if (d > 16777216.0f) d = 16777216.0f;
        float r = 1.0f / d;
        if (bits(div_by_recip(x, d, r)) != bits(x / d)) ++bad;
        ++n;
    }
    printf("%ld %ld\n", n, bad);
    return 0;
}
