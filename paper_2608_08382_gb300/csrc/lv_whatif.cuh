// What-if evaluation over (pending request x candidate batch) pairs.
#pragma once
#include "lv_kernels.cuh"
