// Status codes shared by the C ABI and the internal C++ code.
#pragma once
#include "../../include/ndvm.h"
